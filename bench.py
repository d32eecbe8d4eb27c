#!/usr/bin/env python
"""Benchmark of the QuaRTZ W4A4 hot path on FLUX.1-schnell-shaped block linears.

One step = the whole hot path over one batch: for each of the four MM-DiT
block linears (QKV 3072->9216, proj 3072->3072, MLP 3072->12288 and
12288->3072, M = (4096 + 512) tokens x batch 4 = 18432), quantize + LZS-encode
the fp16 activations (Eq. 1, Eq. 2), expand the codes and run the tcgen05
GEMM with its dequant epilogue (Section 4.4).  Weights are encoded, and
their tensor-core operand prepared, once, offline, outside the timed region
(as the paper's PTQ does).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  `value` is W4A4 linear TOPS of the whole job
(2*M*N*K summed over the layers, per step, over the device-timed step
time); the encode GB/s of the quantize kernel is reported beside it.  The
inputs (~0.8 GB of fp16 activations per step) exceed the 129 MB L2, so no
flush is needed between steps.  Multi-GPU runs are independent replicas
(the path shards by token rows with no exchange): weak scaling.

Secondary lines in the same JSON object (N = 1): `configs` times the single
256 x 1152 layer, the quantize / decode sweep over 1M / 16M / 128M elements
at G_s 8 / 16 / 32, the PixArt-Sigma and SDXL layers, and the paper's Table 1
layer sizes (L2 flushed before every repetition); `peaks_measured` holds the
fp32-pipe and FP8 tensor rates measured in the same run, the roofline
denominators beside the derived and MEASURED_PEAKS.json figures.
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
sys.path.insert(0, ROOT)

METRIC = "QuaRTZ W4A4 linear TOPS (% of roofline); LZS encode GB/s (% of HBM peak)"
GROUP_Q, GROUP_S = 64, 16
FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS = 6800.0, 1900.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=300)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    p.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline leg")
    p.add_argument("--no-fused", action="store_true", help="skip the fused activation-path leg")
    p.add_argument("--scales", choices=["group64", "per-row"], default="group64",
                   help="group64: 64-wide groups along K (Appendix C, the default workload); "
                        "per-row: one scale per token row and per output channel (group_q = K)")
    p.add_argument("--compare-algos", action="store_true",
                   help="also time the three GEMM algorithms (tcgen05, simt, shift) on each layer")
    p.add_argument("--layers", default="", help="comma-separated subset of layer names (profiling)")
    p.add_argument("--no-attention", dest="attention", action="store_false",
                   help="skip the attention decode step leg (Appendix D, Table 6: heads x 128, "
                        "G_s 8/16/32, a 4096-token encoded cache, batch 16)")
    p.add_argument("--no-configs", dest="configs", action="store_false",
                   help="skip the secondary lines: configs 0-3 (single 1152 layer, encode/decode sweep, "
                        "PixArt and SDXL layers) and the Table 1 layer sizes")
    p.add_argument("--no-llm", dest="llm", action="store_false",
                   help="skip the LLM-variant leg (Section 5: 16-bit codes straight to 4 bits, "
                        "G_s = 8, LLaMA-2-7B block linears)")
    return p.parse_args()


FALLBACK_SM_MHZ = 2070.0
# The GEMM's tensor-core work is FP8 E4M3 (kind::f8f6f4): its peak is the
# measured bf16 peak times the nominal dense FP8 : BF16 ratio (4.5 : 2.25).
FP8_OVER_BF16 = 2.0
# FP32 pipe: 128 lanes per SM, one multiply or fused multiply-add per lane per
# cycle (a paired f32x2 instruction occupies two lanes' worth).
FP32_LANES_PER_SM = 128


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return (float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d.get("sm_max_mhz", FALLBACK_SM_MHZ)),
                "measured")
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, FALLBACK_SM_MHZ, "fallback"


def gemm_source_hash():
    """sha256 (first 16 hex) of the tcgen05 GEMM's source: its section of
    csrc/linear.cu (from the "2. tcgen05 GEMM" banner to the "3. SIMT GEMM"
    banner) plus csrc/ptx.cuh."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_2509_26436_gb300", "csrc")
    with open(os.path.join(csrc, "linear.cu")) as fh:
        src = fh.read()
    section = src[src.index("// 2. tcgen05 GEMM"):src.index("// 3. SIMT GEMM")]
    h = hashlib.sha256(section.encode())
    with open(os.path.join(csrc, "ptx.cuh"), "rb") as fh:
        h.update(fh.read())
    return h.hexdigest()[:16]


def gemm_traffic():
    """DRAM bytes per GEMM launch from the committed ncu summary, if it was
    taken on the GEMM source as it is now (else None)."""
    try:
        with open(os.path.join(ROOT, "profiles", "gemm_tcgen05_flux_block.md")) as fh:
            kv = dict(line.split(": ", 1) for line in fh if line.startswith(("gemm_source_sha16", "dram_bytes")))
    except OSError:
        return None
    if kv.get("gemm_source_sha16", "").strip() != gemm_source_hash():
        return None
    return float(kv["dram_bytes_per_launch"])


def max_over_ranks(t, world, device=None):
    """The slowest rank's time: the whole job finishes when its last rank does."""
    if world <= 1:
        return t
    import torch
    import torch.distributed as dist
    x = torch.tensor([t], dtype=torch.float64, device=device)
    dist.all_reduce(x, op=dist.ReduceOp.MAX)
    return float(x.item())


def host_link_gbs(torch, dev, mib=256, reps=3):
    """Pinned host <-> device copy rates (GB/s): H2D alone, D2H alone and the
    two directions at once on two streams; best of `reps`."""
    n = mib << 20
    h_in = torch.empty(n, dtype=torch.uint8).pin_memory()
    h_out = torch.empty(n, dtype=torch.uint8).pin_memory()
    d_in = torch.empty(n, dtype=torch.uint8, device=dev)
    d_out = torch.zeros(n, dtype=torch.uint8, device=dev)
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    best = {"h2d": 0.0, "d2h": 0.0, "both": 0.0}
    for _ in range(reps):
        for key in best:
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            if key in ("h2d", "both"):
                with torch.cuda.stream(s1):
                    d_in.copy_(h_in, non_blocking=True)
            if key in ("d2h", "both"):
                with torch.cuda.stream(s2):
                    h_out.copy_(d_out, non_blocking=True)
            torch.cuda.synchronize()
            dt = time.perf_counter() - t0
            moved = n * (2 if key == "both" else 1)
            best[key] = max(best[key], moved / dt / 1e9)
    return best


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def layer_config(layers, per_row=False):
    return {"workload": "flux1_schnell_mmdit_block_linears", "tokens": layers[0].M,
            "layers": [f"{l.name}:{l.K}->{l.N}" for l in layers],
            "group_q": "K (per-token x per-channel)" if per_row else GROUP_Q,
            "group_s": GROUP_S, "mode": "symmetric", "out": "f16",
            "inputs": "seeded synthetic Laplace(0,0.05), 0.1% channels x50; weights N(0,0.02)",
            "l2": "activations per step 0.8 GB > 129 MB L2, no flush"}


def select_layers(all_layers, names):
    if not names:
        return list(all_layers)
    want = names.split(",")
    sel = [l for l in all_layers if l.name in want]
    if len(sel) != len(want):
        raise SystemExit(f"unknown layer in {names}; have {[l.name for l in all_layers]}")
    return sel


def encode_bytes_per_elem(gs=GROUP_S, gq=GROUP_Q):
    """Algorithmic HBM bytes of the encoder per element: fp16 in, 4-bit code,
    one FLAG byte per G_s, one fp16 scale per group_q (symmetric)."""
    return 2.0 + 0.5 + 1.0 / gs + 2.0 / gq


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.p = None

    def __enter__(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}",
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.p is not None:
            time.sleep(0.15)
            self.p.terminate()
            self.p.wait()

    def summary(self, bus_id=None):
        self.f.flush()
        self.f.seek(0)
        rows = [[c.strip() for c in line.split(",")] for line in self.f if line.count(",") >= 9]
        os.unlink(self.f.name)
        if bus_id:
            mine = [r for r in rows if r[1].lower().endswith(bus_id.lower()[-12:])]
            rows = mine or rows
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        idx = {r[0] for r in rows}
        if len(idx) > 1:
            rows = [r for r in rows if r[0] == str(self.dev)] or rows
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        smax = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[6:10]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": reasons,
                "samples": len(rows),
                "power_w_max": max((float(r[4]) for r in rows
                                    if r[4].replace(".", "").isdigit()), default=None)}


# --------------------------------------------------------------------------
# CPU oracle baseline (a bounded sample of the same workload)
# --------------------------------------------------------------------------
ORACLE_ROWS = 256


def cpu_model():
    """The host CPU's model name (/proc/cpuinfo, else lscpu, else the ISA)."""
    try:
        with open("/proc/cpuinfo") as fh:
            for line in fh:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    import platform
    return platform.machine()


def oracle_setup(layers, rows_per_layer, xs=None, ws=None, per_row=False):
    """Encode every layer's weights with the oracle (before timing, as the
    GPU path does) and pick `rows_per_layer` evenly spaced token rows."""
    import numpy as np

    import oracle as O
    enc_w, xa_s = [], []
    for i, l in enumerate(layers):
        w = ws[i] if ws is not None else l.weights()
        enc_w.append(O.encode(w, l.K if per_row else GROUP_Q, GROUP_S))
        x = xs[i] if xs is not None else l.activations()
        sel = np.linspace(0, l.M - 1, rows_per_layer).astype(np.int64)
        xa_s.append(np.ascontiguousarray(x[sel]))
    return enc_w, xa_s


def oracle_step(layers, enc_w, xa_s, threads, per_row=False):
    """One sampled step of the oracle: encode (Eq. 1 + Eq. 2) of the sampled
    rows and the W4A4 linear for them, every output channel of every layer.
    The rows of a layer are split into `threads` contiguous chunks run on
    host threads (the oracle's C functions release the GIL).  Returns
    (seconds, ops)."""
    import concurrent.futures as cf

    import numpy as np

    import oracle as O

    def work(l, x, ew):
        ea = O.encode(x, l.K if per_row else GROUP_Q, GROUP_S)
        O.linear(ea, ew)

    t0 = time.perf_counter()
    ops = 0
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        futs = []
        for l, x, ew in zip(layers, xa_s, enc_w):
            for chunk in np.array_split(np.arange(x.shape[0]), threads):
                if chunk.size:
                    futs.append(ex.submit(work, l, np.ascontiguousarray(x[chunk]), ew))
            ops += 2 * x.shape[0] * ew.rows * l.K
        for f in futs:
            f.result()
    return time.perf_counter() - t0, ops


def oracle_sample_desc(rows, threads):
    return (f"{rows} evenly spaced token rows x all output channels of each of the 4 FLUX block linears "
            f"per step (encode + linear), plain C oracle on {threads} host threads (rows split in "
            "contiguous chunks; each thread's call decodes the layer's weights, as the oracle does), "
            "weights encoded before timing")


def oracle_configs(inputs, threads):
    """The oracle on configs 0-3, context for their GPU lines: config 0 in
    full and config 1's encode (1M and 16M elements) on one host thread,
    configs 2 and 3 on ORACLE_ROWS evenly spaced rows per layer on `threads`
    host threads (encode + linear, weights encoded before timing)."""
    import oracle as O
    out = {}
    l0 = inputs.CONFIG0
    enc_w, xa = oracle_setup(l0, l0[0].M)
    t, ops = oracle_step(l0, enc_w, xa, 1)
    out["config0"] = {"TOPS": ops / t / 1e12, "seconds": t, "threads": 1,
                      "sample": "the whole layer (256 x 1152 -> 1152), encode + linear"}
    for key, layers in (("config2", inputs.CONFIG2), ("config3", inputs.CONFIG3)):
        enc_w, xa = oracle_setup(layers, ORACLE_ROWS)
        t, ops = oracle_step(layers, enc_w, xa, threads)
        out[key] = {"TOPS": ops / t / 1e12, "seconds": t, "threads": threads,
                    "sample": f"{ORACLE_ROWS} evenly spaced rows x all output channels of every layer, "
                              "encode + linear"}
    enc = []
    for rows in (256, 4096):
        x = inputs.mixture_activations(rows, 4096, seed=inputs.seed_for(1, 0))
        t0 = time.perf_counter()
        O.encode(x, GROUP_Q, GROUP_S)
        t = time.perf_counter() - t0
        n = rows * 4096
        enc.append({"elements": n, "seconds": t,
                    "gbs": n * (2 + 0.5 + 1 / GROUP_S + 2 / GROUP_Q) / t / 1e9})
    out["config1"] = {"threads": 1, "group_s": GROUP_S, "encode": enc,
                      "sample": "quantize + LZS encode of the sweep's 1M and 16M-element tensors"}
    return out


def run_reference(args):
    from paper_2509_26436_gb300 import inputs
    rank, world, _ = dist_env()
    if rank != 0:
        return
    layers = select_layers(inputs.CONFIG4, args.layers)
    threads = os.cpu_count() or 1
    enc_w, xa_s = oracle_setup(layers, ORACLE_ROWS)
    times = []
    total_ops = 0
    for i in range(args.warmup + args.steps):
        t, ops = oracle_step(layers, enc_w, xa_s, threads)
        if i >= args.warmup:
            times.append(t)
            total_ops = ops
    t_step = sum(times) / len(times)
    value = total_ops / t_step / 1e12
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_step * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64/f64",
        "data": "synthetic", "config": layer_config(layers),
        "cpu_baseline": {"value": value, "unit": "TOPS", "cores": threads, "host_cores": os.cpu_count(),
                         "cpu_model": cpu_model(), "kind": "oracle",
                         "sample": oracle_sample_desc(ORACLE_ROWS, threads)},
        "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# --------------------------------------------------------------------------
# roofline denominators measured in this run
# --------------------------------------------------------------------------
def measure_peaks(torch, Q, dev, n_sm):
    """Rates of the two pipes the GEMM uses, measured here (CUDA events, best
    of several launches, nothing else running):
      fp32_pipe   the paired fp32 multiply / fused multiply-add probe of
                  libquartz (8 CTAs of 256 threads per SM), fp32 lane
                  operations per second;
      fp8_cublas  cuBLASLt FP8 E4M3 GEMM 8192^3 through torch._scaled_mm
                  (the library peak, measured like the bf16 peak in
                  MEASURED_PEAKS.json), FLOP/s;
      fp8_tcgen05 libquartz's MMA probe: back-to-back tcgen05 kind::f8f6f4
                  M128 N256 K32 from shared memory, one CTA per SM (the
                  GEMM's own instruction and shape), FLOP/s."""
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    stream = torch.cuda.current_stream()

    def best(fn, reps):
        fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            e0, e1 = ev(), ev()
            e0.record(stream)
            work = fn()
            e1.record(stream)
            ts.append((e0, e1, work))
        torch.cuda.synchronize()
        return max(w / (a.elapsed_time(b) / 1e3) for a, b, w in ts)

    out = {}
    sink = torch.empty(n_sm * 8 * 256, dtype=torch.float32, device=dev)
    out["fp32_pipe_tops"] = best(lambda: Q.probe_fp32_pipe(n_sm * 8, 20000, sink), 5) / 1e12
    out["fp8_tcgen05_probe_tflops"] = best(lambda: Q.probe_mma_f8(n_sm, 20000), 5) / 1e12
    assert Q.device_status() == 0
    try:
        n = 8192
        g = torch.Generator(device=dev).manual_seed(1)
        a = (torch.rand((n, n), generator=g, device=dev) - 0.5).to(torch.float8_e4m3fn)
        b = (torch.rand((n, n), generator=g, device=dev) - 0.5).to(torch.float8_e4m3fn)
        one = torch.ones((), dtype=torch.float32, device=dev)

        def mm():
            torch._scaled_mm(a, b.t(), one, one, out_dtype=torch.bfloat16)
            return 2 * n ** 3
        out["fp8_cublas_tflops"] = best(mm, 10) / 1e12
        del a, b
    except (RuntimeError, AttributeError, TypeError) as exc:
        out["fp8_cublas_tflops"] = None
        out["fp8_cublas_error"] = str(exc).splitlines()[0][:160]
    return out


# --------------------------------------------------------------------------
# our path
# --------------------------------------------------------------------------
def run_ours(args):
    import numpy as np
    import torch

    import paper_2509_26436_gb300 as Q
    from paper_2509_26436_gb300 import inputs

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    hbm_peak, bf16_peak, sm_mhz, peak_src = peaks()
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    meas = measure_peaks(torch, Q, dev, n_sm)
    if meas.get("fp8_cublas_tflops"):
        fp8_peak = meas["fp8_cublas_tflops"]                          # TFLOP/s
        fp8_src = "measured in this run: cuBLASLt FP8 E4M3 GEMM 8192^3 (torch._scaled_mm), best of 10"
    else:
        fp8_peak = bf16_peak * FP8_OVER_BF16
        fp8_src = f"{peak_src} bf16 burst {bf16_peak} x {FP8_OVER_BF16} (nominal FP8 : BF16)"
    alu_peak = n_sm * FP32_LANES_PER_SM * sm_mhz * 1e6 / 1e12         # T fp32-pipe lane ops/s
    layers = select_layers(inputs.CONFIG4, args.layers)

    # ---- inputs (seeded, host) -> pinned host + device ---------------------
    xs = [l.activations() for l in layers]
    ws = [l.weights() for l in layers]
    x_host = [torch.from_numpy(x).pin_memory() for x in xs]
    x_dev = [h.to(dev) for h in x_host]
    per_row = args.scales == "per-row"
    gq = [l.K if per_row else GROUP_Q for l in layers]
    enc_w = [Q.encode_weights(torch.from_numpy(w).to(dev), group_s=GROUP_S, group_q=g) for w, g in zip(ws, gq)]
    # weights are encoded and their tensor-core operand prepared once, offline
    prep_w = [Q.prepare_weights(w) for w in enc_w]
    enc_a = [Q.empty_encoded(l.M, l.K, Q.Params(g, GROUP_S), dev) for l, g in zip(layers, gq)]
    y_dev = [torch.empty((l.M, l.N), dtype=torch.float16, device=dev) for l in layers]
    ws_bytes = max(Q.linear_workspace_size(l.M, l.N, l.K) for l in layers)
    workspace = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    assert Q.device_status() == 0

    nl = len(layers)
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731

    def step(rec=None):
        for i in range(nl):
            if rec is not None:
                rec["q"][i][0].record(stream)
            Q.quantize(x_dev[i], out=enc_a[i], group_s=GROUP_S, group_q=gq[i])
            if rec is not None:
                rec["q"][i][1].record(stream)
            Q.linear(enc_a[i], enc_w[i], out=y_dev[i], workspace=workspace, w_prepared=prep_w[i],
                     gemm_events=None if rec is None else rec["g"][i])

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    assert Q.device_status() == 0

    # per-kernel durations: every step records events around the quantize
    # kernel and around the GEMM kernel of every layer
    recs = [{"q": [(ev(), ev()) for _ in range(nl)], "g": [(ev(), ev()) for _ in range(nl)]}
            for _ in range(args.steps)]
    bus = None
    try:
        bus = torch.cuda.get_device_properties(dev).pci_bus_id
    except AttributeError:
        pass
    t0, t1 = ev(), ev()
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0.record(stream)
        for k in range(args.steps):
            step(recs[k])
        t1.record(stream)
        torch.cuda.synchronize()
    barrier()
    clocks = clk.summary(bus)
    status = Q.device_status()
    assert status == 0, f"device status {status}"
    t_step = t0.elapsed_time(t1) / 1e3 / args.steps
    t_step = max_over_ranks(t_step, world, dev)

    ops_step = sum(l.ops for l in layers)
    value = world * ops_step / t_step / 1e12
    gemm_ms = [statistics.mean(r["g"][i][0].elapsed_time(r["g"][i][1]) for r in recs)
               for i in range(nl)]
    quant_ms = [statistics.mean(r["q"][i][0].elapsed_time(r["q"][i][1]) for r in recs)
                for i in range(nl)]
    t_gemm = sum(gemm_ms) / 1e3
    gemm_tflops = sum(l.ops for l in layers) / t_gemm / 1e12
    # dequant epilogue: one fp32 multiply and one fused multiply-add per
    # output element and 64-wide group (y += s_a * (s_w * P_g)); with per-row
    # scales one float add and one integer add per output and 256 of K
    if per_row:
        epi_ops = sum(2 * l.M * l.N * -(-l.K // 256) for l in layers)
    else:
        epi_ops = sum(2 * l.M * l.N * (l.K // GROUP_Q) for l in layers)
    gemm_alu = epi_ops / t_gemm / 1e12
    t_floor_tensor = sum(l.ops for l in layers) / (fp8_peak * 1e12)
    t_floor_alu = epi_ops / (alu_peak * 1e12)
    elems = sum(l.M * l.K for l in layers)
    enc_bytes = sum(l.M * l.K * encode_bytes_per_elem(GROUP_S, g) for l, g in zip(layers, gq))
    enc_gbs = enc_bytes / (sum(quant_ms) / 1e3) / 1e9
    # quantize; prepare (activations); GEMM; and, where the GEMM splits its
    # last wave of tiles along K, the kernel that adds the parts
    gemm_launches = [Q.linear_launch_count(l.M, l.N, l.K, Q.Params(g, GROUP_S)) for l, g in zip(layers, gq)]
    launches_per_step = nl + sum(gemm_launches)

    alu_view = {"achieved": gemm_alu, "unit": "Top/s", "peak": alu_peak, "frac": gemm_alu / alu_peak,
                "peak_source": f"derived: {n_sm} SMs x {FP32_LANES_PER_SM} fp32 lanes x "
                               f"{sm_mhz:.0f} MHz ({peak_src} max SM clock)",
                "peak_measured": meas["fp32_pipe_tops"],
                "frac_of_measured": gemm_alu / meas["fp32_pipe_tops"],
                "peak_measured_source": "measured in this run: paired fp32 mul/fma probe "
                                        "(quartz_probe_fp32_pipe), best of 5",
                "work": ("1 fp32 add + 1 int32 add per output per 256 of K" if per_row else
                         "2 fp32 ops (multiply + fused multiply-add) per output per 64-wide group")}
    tensor_view = {"achieved": gemm_tflops, "unit": "TFLOP/s", "peak": fp8_peak, "frac": gemm_tflops / fp8_peak,
                   "peak_source": fp8_src,
                   "tcgen05_probe_peak": meas["fp8_tcgen05_probe_tflops"],
                   "frac_of_tcgen05_probe": gemm_tflops / meas["fp8_tcgen05_probe_tflops"],
                   "work": "2 M N K FP8 MMA flops"}
    bound = "alu" if t_floor_alu >= t_floor_tensor else "tensor"
    main, other = (alu_view, tensor_view) if bound == "alu" else (tensor_view, alu_view)
    roofline = {"bound": bound, **main, "traffic": None if per_row else gemm_traffic(),
                "kernel": "gemm_tcgen05_kernel",
                "tensor" if bound == "alu" else "alu": other,
                "floors_ms": {"alu": t_floor_alu * 1e3, "tensor": t_floor_tensor * 1e3},
                "per_layer_ms": gemm_ms}

    # ---- fused activation path (quartz_linear_f16: encode into the operand) -
    fused = None
    if not args.no_fused and not per_row:
        def fused_step():
            for i in range(nl):
                Q.linear_f16(x_dev[i], enc_w[i], out=y_dev[i], workspace=workspace, w_prepared=prep_w[i])

        for _ in range(args.warmup):
            fused_step()
        torch.cuda.synchronize()
        barrier()
        f0, f1 = ev(), ev()
        f0.record(stream)
        for _ in range(args.steps):
            fused_step()
        f1.record(stream)
        torch.cuda.synchronize()
        barrier()
        assert Q.device_status() == 0
        tf = f0.elapsed_time(f1) / 1e3 / args.steps
        tf = max_over_ranks(tf, world, dev)
        fused = {"value": world * ops_step / tf / 1e12, "unit": "TOPS", "ms_per_step": tf * 1e3,
                 "path": "quartz_linear_f16_ex per layer with prepared weights (activations encoded "
                         "straight into the GEMM operand; bit-identical to quantize + linear)",
                 "gpu_launches": sum(gemm_launches) * args.steps}

    # ---- GEMM algorithms side by side (optional) ----------------------------
    algos = None
    if args.compare_algos:
        algos = {}
        for name, algo in (("tcgen05", Q.ALGO_TCGEN05), ("simt", Q.ALGO_SIMT), ("shift", Q.ALGO_SHIFT)):
            per = []
            for i in range(nl):
                Q.quantize(x_dev[i], out=enc_a[i], group_s=GROUP_S, group_q=gq[i])
                Q.linear(enc_a[i], enc_w[i], out=y_dev[i], workspace=workspace, algo=algo)
                evs = [(ev(), ev()) for _ in range(3)]
                for e in evs:
                    Q.linear(enc_a[i], enc_w[i], out=y_dev[i], workspace=workspace, algo=algo, gemm_events=e)
                torch.cuda.synchronize()
                ms = statistics.median(e[0].elapsed_time(e[1]) for e in evs)
                per.append({"layer": layers[i].name, "ms": ms, "TOPS": layers[i].ops / ms / 1e9})
            algos[name] = per
        algos["tuning"] = ("tcgen05: the tuned product kernel; simt and shift: plain 64 x 64-tile CUDA-core "
                           "kernels, untuned")
        assert Q.device_status() == 0

    # ---- LLM variant (optional) ---------------------------------------------
    llm = run_llm_variant(args, Q, inputs, dev, n_sm, sm_mhz, peak_src, fp8_peak, fp8_src) if args.llm else None
    attn = run_attention(args, Q, inputs, dev, hbm_peak, peak_src) if args.attention else None
    configs = (run_configs(args, torch, Q, inputs, dev, hbm_peak, alu_peak, fp8_peak)
               if args.configs and world == 1 and not per_row else None)

    # ---- end to end through the public API with host buffers ---------------
    # Each (step, layer) unit copies its activations from pinned host memory,
    # encodes them, runs the linear layer and copies the fp16 output back to
    # pinned host memory.  Copies run on their own streams, double-buffered,
    # so the H2D of the next unit and the D2H of the previous one overlap the
    # compute of the current one; the timed region spans all three streams.
    e2e = None
    if not args.no_e2e:
        y_host = [torch.empty((l.M, l.N), dtype=torch.float16).pin_memory() for l in layers]
        x_buf = [[torch.empty_like(x_dev[i]) for i in range(nl)] for _ in range(2)]
        y_buf = [[torch.empty_like(y_dev[i]) for i in range(nl)] for _ in range(2)]
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        e_steps = max(20, min(args.steps, 50))

        def e2e_run(n_steps, compute=True):
            # unit u = (step, layer) uses buffer set u % 2 of its layer, last
            # used by unit u - 2 nl: its H2D waits only for that unit's encode
            # and its compute only for that unit's D2H, so compute can run up
            # to 2 nl - 1 units ahead of the slower D2H stream.  compute=False
            # issues the same copies and events without the kernels (the
            # control that shows what the host link alone allows)
            loaded, consumed, computed, drained = {}, {}, {}, {}
            units = [(k, i) for k in range(n_steps) for i in range(nl)]
            back = 2 * nl
            for u, (k, i) in enumerate(units):
                p = (u // nl) % 2
                with torch.cuda.stream(s_in):
                    if u >= back:
                        s_in.wait_event(consumed[u - back])
                    x_buf[p][i].copy_(x_host[i], non_blocking=True)
                    loaded[u] = torch.cuda.Event()
                    loaded[u].record(s_in)
                stream.wait_event(loaded[u])
                if compute:
                    Q.quantize(x_buf[p][i], out=enc_a[i], group_s=GROUP_S, group_q=gq[i])
                consumed[u] = torch.cuda.Event()
                consumed[u].record(stream)
                if u >= back:
                    stream.wait_event(drained[u - back])
                if compute:
                    Q.linear(enc_a[i], enc_w[i], out=y_buf[p][i], workspace=workspace, w_prepared=prep_w[i])
                computed[u] = torch.cuda.Event()
                computed[u].record(stream)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(computed[u])
                    y_host[i].copy_(y_buf[p][i], non_blocking=True)
                    drained[u] = torch.cuda.Event()
                    drained[u].record(s_out)
            stream.wait_event(drained[len(units) - 1])

        e2e_run(2)
        e2e_run(2, compute=False)
        torch.cuda.synchronize()

        def timed_rep(compute):
            barrier()
            a0, a1 = ev(), ev()
            a0.record(stream)
            s_in.wait_stream(stream)
            e2e_run(e_steps, compute)
            a1.record(stream)
            torch.cuda.synchronize()
            barrier()
            return max_over_ranks(a0.elapsed_time(a1) / 1e3 / e_steps, world, dev)

        # five timed repetitions of e_steps steps each, every one followed by
        # the same copies without the kernels; the median is the value.  The
        # host link itself alternates between two rates from one repetition
        # to the next (copies alone: about 5.8 or 6.8-7.0 ms per FLUX step),
        # so the spread of the repetitions is the link's; the ratio to the
        # copies alone is what the pipeline adds.
        reps, copy_reps = [], []
        for _ in range(5):
            reps.append(timed_rep(True))
            copy_reps.append(timed_rep(False))
        te = statistics.median(reps)
        tc = statistics.median(copy_reps)
        h2d = sum(x.numel() * 2 for x in x_host)
        d2h = sum(l.M * l.N * 2 for l in layers)
        link = host_link_gbs(torch, dev)
        floor = max(h2d / (link["h2d"] * 1e9), d2h / (link["d2h"] * 1e9), (h2d + d2h) / (link["both"] * 1e9))
        e2e = {"value": world * ops_step / te / 1e12, "unit": "TOPS",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e_steps,
               "ms_per_step": te * 1e3, "repetitions": len(reps),
               "ms_per_step_reps": [r * 1e3 for r in reps],
               "spread": (max(reps) - min(reps)) / te,
               "copies_alone": {"ms_per_step": tc * 1e3, "ms_per_step_reps": [r * 1e3 for r in copy_reps],
                                "e2e_over_copies": te / tc,
                                "what": "the same H2D / D2H copies and events with no kernels, timed after "
                                        "each end-to-end repetition"},
               "overlap": "H2D / compute / D2H on three streams, two buffer sets per layer (compute up to "
                          "2 x layers - 1 units ahead of the D2H stream)",
               "roofline": {"bound": "host link", "link_gbs_measured": link,
                            "floor_ms": floor * 1e3, "frac": floor / te,
                            "work": "the step's H2D and D2H bytes at the link rates measured here "
                                    "(pinned 256 MiB copies, each direction alone and both at once)"}}

    # ---- CPU oracle baseline (rank 0 only, N = 1) ---------------------------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        threads = os.cpu_count() or 1
        enc_w_o, xa_o = oracle_setup(layers, ORACLE_ROWS, xs, ws, per_row=per_row)
        tt, oo = 0.0, 0
        for _ in range(3):
            t, ops = oracle_step(layers, enc_w_o, xa_o, threads, per_row=per_row)
            tt, oo = tt + t, oo + ops
        cpu = {"value": oo / tt / 1e12, "unit": "TOPS", "cores": threads, "host_cores": os.cpu_count(),
               "cpu_model": cpu_model(), "kind": "oracle",
               "sample": oracle_sample_desc(ORACLE_ROWS, threads) + f"; 3 steps, {tt:.1f} s"}
        if args.configs and not per_row:
            from paper_2509_26436_gb300 import inputs as inp
            cpu["configs"] = oracle_configs(inp, threads)

    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    if rank != 0:
        return
    out = {
        "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_step * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "e4m3/f32", "data": "synthetic",
        "config": layer_config(layers, per_row),
        "roofline": roofline,
        "encode": {"kernel": "quantize_kernel", "gbs": enc_gbs, "peak_gbs": hbm_peak,
                   "frac": enc_gbs / hbm_peak, "bytes_per_elem": enc_bytes / elems,
                   "per_layer_ms": quant_ms, "peak_source": peak_src},
        "clocks": clocks,
        "gpu_launches": launches_per_step * args.steps,
        "fused": fused,
        "gemm_algos": algos,
        "llm_variant": llm,
        "attention": attn,
        "configs": configs,
        "peaks_measured": meas,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    print(json.dumps(out), flush=True)


# --------------------------------------------------------------------------
# configs 0-3 and the paper's Table 1 layer sizes (secondary bench lines)
# --------------------------------------------------------------------------
L2_FLUSH_BYTES = 256 << 20   # read before every timed repetition (> 129 MB L2)
CONFIG_REPS = 10


def gemm_roofline(layers, gemm_ms, alu_peak, fp8_peak):
    """Both floors of the tcgen05 GEMM for `layers` at the given per-layer
    GEMM times: the fp32 pipe (2 ops per output and 64-group) and the FP8
    tensor pipe (2 M N K)."""
    t = sum(gemm_ms) / 1e3
    epi = sum(2 * l.M * l.N * (l.K // GROUP_Q) for l in layers)
    ops = sum(l.ops for l in layers)
    alu, ten = epi / t / 1e12, ops / t / 1e12
    return {"bound": "alu", "achieved": alu, "peak": alu_peak, "unit": "Top/s", "frac": alu / alu_peak,
            "tensor": {"achieved": ten, "peak": fp8_peak, "unit": "TFLOP/s", "frac": ten / fp8_peak}}


def time_linear_layers(torch, Q, dev, layers, xs, ws, flush, reps=CONFIG_REPS, group_s=GROUP_S):
    """Per layer: quantize + linear (prepared weights), L2 flushed before each
    repetition; CUDA events around the quantize kernel, the GEMM (+ tail
    combine) and the whole layer.  Returns per-layer medians in ms."""
    stream = torch.cuda.current_stream()
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    out = []
    for l, x, w in zip(layers, xs, ws):
        xd = torch.from_numpy(x).to(dev)
        ew = Q.encode_weights(torch.from_numpy(w).to(dev), group_s=group_s)
        pw = Q.prepare_weights(ew)
        ea = Q.empty_encoded(l.M, l.K, Q.Params(GROUP_Q, group_s), dev)
        y = torch.empty((l.M, l.N), dtype=torch.float16, device=dev)
        wsb = torch.empty(max(Q.linear_workspace_size(l.M, l.N, l.K, ea.params), 16), dtype=torch.uint8,
                          device=dev)
        for _ in range(3):
            Q.quantize(xd, out=ea, group_s=group_s)
            Q.linear(ea, ew, out=y, workspace=wsb, w_prepared=pw)
        recs = []
        for _ in range(reps):
            flush()
            e = [ev() for _ in range(5)]
            e[0].record(stream)
            Q.quantize(xd, out=ea, group_s=group_s)
            e[1].record(stream)
            Q.linear(ea, ew, out=y, workspace=wsb, w_prepared=pw, gemm_events=(e[2], e[3]))
            e[4].record(stream)
            recs.append(e)
        torch.cuda.synchronize()
        assert Q.device_status() == 0
        med = lambda i, j: statistics.median(r[i].elapsed_time(r[j]) for r in recs)  # noqa: E731
        out.append({"layer": l.name, "M": l.M, "N": l.N, "K": l.K, "ms": med(0, 4), "quantize_ms": med(0, 1),
                    "gemm_ms": med(2, 3), "TOPS": l.ops / med(0, 4) / 1e9,
                    "gemm_TOPS": l.ops / med(2, 3) / 1e9,
                    "launches": 1 + Q.linear_launch_count(l.M, l.N, l.K, ea.params)})
        del xd, ew, pw, ea, y, wsb
    return out


def run_encode_sweep(torch, Q, inputs, dev, hbm_peak, flush, reps=CONFIG_REPS):
    """Config 1: quantize + LZS encode and decode (quartz_dequantize) of
    1M / 16M / 128M fp16 elements ([256 | 4096 | 32768, 4096]) at G_s 8 / 16 /
    32.  Throughput: back-to-back launches over distinct row slices of one
    128M-element tensor (and of one encoded tensor and one output tensor),
    so that every launch reads and writes memory no earlier launch of the
    cycle touched: 256 MB of inputs per cycle of slices (128 slices of 1M, 8
    of 16M, the whole 128M), far above the 129 MB L2; CUDA events around
    the whole sequence.  Latency: one launch after a 256 MiB L2 flush."""
    stream = torch.cuda.current_stream()
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    K, R_ALL = 4096, 32768
    x_all = torch.from_numpy(inputs.mixture_activations(R_ALL, K, seed=inputs.seed_for(1, 0))).to(dev)
    xhat_all = torch.empty_like(x_all)
    res = []
    for gs in (8, 16, 32):
        e_all = Q.empty_encoded(R_ALL, K, Q.Params(GROUP_Q, gs), dev)

        def enc_slice(i, rows):
            sl = slice(i * rows, (i + 1) * rows)
            return Q.Encoded(e_all.codes[sl], e_all.flags[sl], e_all.scales[sl], None, None, rows, K, e_all.params)

        for rows in (256, 4096, 32768):
            n_sl = R_ALL // rows
            xs = [x_all[i * rows:(i + 1) * rows] for i in range(n_sl)]
            hs = [xhat_all[i * rows:(i + 1) * rows] for i in range(n_sl)]
            es = [enc_slice(i, rows) for i in range(n_sl)]
            launches = max(20, n_sl)
            for i in range(min(n_sl, 4)):
                Q.quantize(xs[i], out=es[i], group_s=gs)
                Q.dequantize(es[i], out=hs[i])
            times = {}
            for kind in ("encode", "decode"):
                # the launches are captured in a CUDA graph so that the host's
                # per-call cost does not starve the GPU between small kernels
                g = torch.cuda.CUDAGraph()
                side = torch.cuda.Stream(dev)
                side.wait_stream(stream)
                with torch.cuda.stream(side):
                    with torch.cuda.graph(g, stream=side):
                        for i in range(launches):
                            if kind == "encode":
                                Q.quantize(xs[i % n_sl], out=es[i % n_sl], group_s=gs)
                            else:
                                Q.dequantize(es[i % n_sl], out=hs[i % n_sl])
                stream.wait_stream(side)
                g.replay()
                torch.cuda.synchronize()
                reps_t = []
                for _ in range(3):
                    a, b = ev(), ev()
                    a.record(stream)
                    g.replay()
                    b.record(stream)
                    reps_t.append((a, b))
                torch.cuda.synchronize()
                times[kind] = statistics.median(a.elapsed_time(b) for a, b in reps_t) / launches
                del g
            lat = {"encode": [], "decode": []}
            for _ in range(reps):
                for kind in ("encode", "decode"):
                    flush()
                    a, b = ev(), ev()
                    a.record(stream)
                    if kind == "encode":
                        Q.quantize(xs[0], out=es[0], group_s=gs)
                    else:
                        Q.dequantize(es[0], out=hs[0])
                    b.record(stream)
                    lat[kind].append((a, b))
            torch.cuda.synchronize()
            assert Q.device_status() == 0
            n = rows * K
            enc_b = n * encode_bytes_per_elem(gs, GROUP_Q)
            dec_b = n * (0.5 + 1.0 / gs + 2.0 / GROUP_Q + 2.0)
            ms_e, ms_d = times["encode"], times["decode"]
            res.append({"elements": n, "shape": [rows, K], "group_s": gs, "launches": launches,
                        "encode_us": ms_e * 1e3, "encode_gbs": enc_b / ms_e / 1e6,
                        "encode_frac": enc_b / ms_e / 1e6 / hbm_peak,
                        "decode_us": ms_d * 1e3, "decode_gbs": dec_b / ms_d / 1e6,
                        "decode_frac": dec_b / ms_d / 1e6 / hbm_peak,
                        "encode_latency_us": statistics.median(a.elapsed_time(b) for a, b in lat["encode"]) * 1e3,
                        "decode_latency_us": statistics.median(a.elapsed_time(b) for a, b in lat["decode"]) * 1e3,
                        "note": "latency-bound (2.7 MB moved per launch)" if rows == 256 else "hbm-bound"})
        del e_all
    del x_all, xhat_all
    res.sort(key=lambda r: (r["elements"], r["group_s"]))
    return {"workload": "quantize+LZS encode / decode sweep, fp16 mixture 89% Laplace(0,0.05), "
                        "10% N(0,0.3), 1% U(-8,8)",
            "kernels": "quantize_sym_kernel / dequantize_kernel", "peak_gbs": hbm_peak,
            "encode_bytes": "2 + 1/2 + 1/G_s + 2/64 B per element",
            "decode_bytes": "1/2 + 1/G_s + 2/64 + 2 B per element",
            "l2": "throughput: back-to-back launches (one CUDA graph, replayed 3 times, median) over "
                  "distinct slices, 256 MB of inputs per cycle (> 129 MB L2); latency: one launch after "
                  f"a 256 MiB read of another buffer, median of {reps}",
            "sizes": res}


def run_configs(args, torch, Q, inputs, dev, hbm_peak, alu_peak, fp8_peak):
    """Throughput of configs 0-3 and, as context for the paper's Table 1
    (A100 latencies of 4096^2 / 5120^2 / 8192^2 layers at G_s 8 / 16 / 32, M
    not stated), the same layers at M = 4096 tokens."""
    # L2 flush: read a buffer larger than L2, so that the timed kernel starts
    # with L2 full of clean lines of another tensor (a written buffer would
    # leave dirty lines whose write-back lands inside the timed kernel)
    buf = torch.zeros(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    flush = lambda: torch.sum(buf)  # noqa: E731
    out = {"l2": f"{L2_FLUSH_BYTES >> 20} MiB read before every repetition; medians of {CONFIG_REPS}"}
    for key, layers, desc in (("config0", inputs.CONFIG0, "single W4A4 linear 256 x 1152 -> 1152"),
                              ("config2", inputs.CONFIG2, "PixArt-Sigma block linears, 8192 tokens"),
                              ("config3", inputs.CONFIG3, "SDXL UNet 3x3 convs as im2col GEMMs, batch 2")):
        xs = [l.activations() for l in layers]
        ws = [l.weights() for l in layers]
        per = time_linear_layers(torch, Q, dev, layers, xs, ws, flush)
        t = sum(p["ms"] for p in per)
        out[key] = {"workload": desc, "group_q": GROUP_Q, "group_s": GROUP_S, "mode": "symmetric", "out": "f16",
                    "TOPS": sum(l.ops for l in layers) / t / 1e9, "ms_per_step": t,
                    "layers": per,
                    "roofline": gemm_roofline(layers, [p["gemm_ms"] for p in per], alu_peak, fp8_peak)}
    out["config1"] = run_encode_sweep(torch, Q, inputs, dev, hbm_peak, flush)
    # Table 1 context: the paper reports 0.189 / 0.184 / 0.176 ms (4096^2),
    # 0.383 / 0.268 / 0.239 ms (5120^2) and 0.468 / 0.327 / 0.313 ms (8192^2)
    # at g8 / g16 / g32 on an A100, M unstated
    paper = {4096: (0.189, 0.184, 0.176), 5120: (0.383, 0.268, 0.239), 8192: (0.468, 0.327, 0.313)}
    rows = []
    for n, ref in paper.items():
        w = inputs.gaussian_weights(n, n, seed=inputs.seed_for(7, n % 97, 1))
        for M in (1024, 4096):
            x = inputs.laplace_activations(M, n, seed=inputs.seed_for(7, n % 97))
            for gs, ref_ms in zip((8, 16, 32), ref):
                l = inputs.Layer(f"table1_{n}", M, n, n, 7, 0)
                p = time_linear_layers(torch, Q, dev, [l], [x], [w], flush, group_s=gs)[0]
                rows.append({"layer": f"{n}x{n}", "M": M, "group_s": gs, "ms": p["ms"], "gemm_ms": p["gemm_ms"],
                             "TOPS": p["TOPS"], "paper_a100_ms": ref_ms})
    out["table1_context"] = {"note": "paper: A100, s4 x s4 -> s32, M not stated (context, not a target; at "
                                     "8192^2 and 0.313 ms, M = 4096 would need 1756 TOPS, above the A100's "
                                     "dense int4 peak, so its M is smaller); here: one GB300, M = 1024 and "
                                     "4096 tokens, quantize + linear per call",
                             "rows": rows}
    del buf
    return out


LLM_GROUP_S = 8


def run_attention(args, Q, inputs, dev, hbm_peak, peak_src):
    """Attention decode step (one query per batch x head over an encoded
    4096-token key / value cache) for each Table 6 setting: heads x 128 and
    G_s in {8, 16, 32}.  Time = CUDA events around quartz_attention_decode
    (split kernel + combine), median of the timed repetitions; roofline =
    algorithmic cache bytes over the measured HBM copy peak."""
    import torch
    B, L, d = inputs.ATTN_BATCH, inputs.ATTN_CONTEXT, inputs.ATTN_DIM
    BHmax = B * max(inputs.ATTN_HEADS)
    xq, xk, xv = inputs.attention_inputs(BHmax, L, seed=inputs.BASE_SEED + 6000)
    xq_d, xk_d, xv_d = (torch.from_numpy(x).to(dev) for x in (xq, xk, xv))
    del xk, xv
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    reps = max(5, min(args.steps, 50))
    out = []
    for heads in inputs.ATTN_HEADS:
        BH = B * heads
        for gs in (8, 16, 32):
            q = Q.quantize(xq_d[:BH].contiguous(), group_s=gs)
            k = Q.quantize(xk_d[:BH * L], group_s=gs)
            v = Q.quantize(xv_d[:BH * L], group_s=gs)
            o = torch.empty((BH, d), dtype=torch.float16, device=dev)
            ws = torch.empty(Q.attention_workspace_size(BH, L), dtype=torch.uint8, device=dev)
            for _ in range(max(3, args.warmup)):
                Q.attention_decode(q, k, v, L, L, d ** -0.5, out=o, workspace=ws)
            torch.cuda.synchronize()
            times = []
            for _ in range(reps):
                e0, e1 = ev(), ev()
                e0.record()
                Q.attention_decode(q, k, v, L, L, d ** -0.5, out=o, workspace=ws)
                e1.record()
                times.append((e0, e1))
            torch.cuda.synchronize()
            assert Q.device_status() == 0
            ms = statistics.median(a.elapsed_time(b) for a, b in times)
            cache_bytes = 2 * BH * L * (d // 2 + d // gs + 2 * (d // GROUP_Q))
            gbs = cache_bytes / (ms / 1e3) / 1e9
            out.append({"heads": heads, "dim": d, "group_s": gs, "batch": B, "context": L, "us": ms * 1e3,
                        "cache_bytes": cache_bytes, "gbs": gbs, "frac": gbs / hbm_peak,
                        "fp16_cache_bytes": 2 * BH * L * d * 2})
            del q, k, v, o, ws
    return {"workload": "attention decode step over an encoded key/value cache (Table 6 settings)",
            "kernels": "attn_decode_kernel + attn_combine_kernel", "peak_gbs": hbm_peak,
            "peak_source": peak_src, "bound": "hbm",
            "bytes": "2 x BH x L x (d/2 codes + d/G_s FLAG bytes + 2 fp16 scales x d/64) per step",
            "inputs": "seeded synthetic N(0,1) q, k, v; 2% of key dims x8; caches > L2 (no flush)",
            "settings": out}


def run_llm_variant(args, Q, inputs, dev, n_sm, sm_mhz, peak_src, fp8_peak, fp8_src):
    """One step = encode (16-bit codes, G_s = 8) + linear of each of the four
    LLaMA-2-7B block linears at 2048 tokens; per-kernel CUDA-event times, for
    the tcgen05 GEMM (E5M2 operands) and the exact accumulator-shift GEMM."""
    import torch
    layers = inputs.CONFIG_LLM
    nl = len(layers)
    x_dev = [torch.from_numpy(l.activations()).to(dev) for l in layers]
    enc_w = [Q.encode_weights(torch.from_numpy(l.weights()).to(dev), group_s=LLM_GROUP_S, code_bits=16)
             for l in layers]
    prep_w = [Q.prepare_weights(w) for w in enc_w]
    enc_a = [Q.empty_encoded(l.M, l.K, Q.Params(GROUP_Q, LLM_GROUP_S, code_bits=16), dev) for l in layers]
    y_dev = [torch.empty((l.M, l.N), dtype=torch.float16, device=dev) for l in layers]
    workspace = torch.empty(max(Q.linear_workspace_size(l.M, l.N, l.K, enc_a[0].params) for l in layers),
                            dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    ops = sum(l.ops for l in layers)
    alu_peak = n_sm * FP32_LANES_PER_SM * sm_mhz * 1e6 / 1e12
    enc_bytes = sum(l.M * l.K * encode_bytes_per_elem(LLM_GROUP_S, GROUP_Q) for l in layers)

    def timed(algo, steps):
        def step(rec=None):
            for i in range(nl):
                if rec is not None:
                    rec[i][0].record(stream)
                Q.quantize(x_dev[i], out=enc_a[i], group_s=LLM_GROUP_S, code_bits=16)
                if rec is not None:
                    rec[i][1].record(stream)
                Q.linear(enc_a[i], enc_w[i], out=y_dev[i], workspace=workspace, algo=algo, w_prepared=prep_w[i],
                         gemm_events=None if rec is None else rec[i][2:])

        for _ in range(max(3, args.warmup)):
            step()
        torch.cuda.synchronize()
        recs = [[(ev(), ev(), ev(), ev()) for _ in range(nl)] for _ in range(steps)]
        t0, t1 = ev(), ev()
        t0.record(stream)
        for k in range(steps):
            step(recs[k])
        t1.record(stream)
        torch.cuda.synchronize()
        assert Q.device_status() == 0
        t_step = t0.elapsed_time(t1) / 1e3 / steps
        gemm_ms = [statistics.mean(r[i][2].elapsed_time(r[i][3]) for r in recs) for i in range(nl)]
        quant_ms = [statistics.mean(r[i][0].elapsed_time(r[i][1]) for r in recs) for i in range(nl)]
        return t_step, gemm_ms, quant_ms

    def timed_fused(steps):
        # the fused activation path: one encoder launch writes the E5M2
        # operand straight from fp16 (bit-identical to the two-call path)
        def step():
            for i in range(nl):
                Q.linear_f16(x_dev[i], enc_w[i], out=y_dev[i], workspace=workspace, w_prepared=prep_w[i])

        for _ in range(max(3, args.warmup)):
            step()
        torch.cuda.synchronize()
        t0, t1 = ev(), ev()
        t0.record(stream)
        for _ in range(steps):
            step()
        t1.record(stream)
        torch.cuda.synchronize()
        assert Q.device_status() == 0
        return t0.elapsed_time(t1) / 1e3 / steps

    t_tc, gemm_tc, quant_ms = timed(Q.ALGO_TCGEN05, max(3, min(args.steps, 50)))
    t_fused = timed_fused(max(3, min(args.steps, 50)))
    t_sh, gemm_sh, _ = timed(Q.ALGO_SHIFT, max(1, min(args.steps, 5)))
    t_gemm = sum(gemm_tc) / 1e3
    epi_ops = sum(2 * l.M * l.N * (l.K // GROUP_Q) for l in layers)
    t_floor_alu, t_floor_tensor = epi_ops / (alu_peak * 1e12), ops / (fp8_peak * 1e12)
    alu_view = {"achieved": epi_ops / t_gemm / 1e12, "peak": alu_peak, "unit": "Top/s",
                "frac": epi_ops / t_gemm / 1e12 / alu_peak,
                "work": "2 fp32 ops (multiply + fused multiply-add) per output per 64-wide group"}
    tensor_view = {"achieved": ops / t_gemm / 1e12, "peak": fp8_peak, "unit": "TFLOP/s",
                   "frac": ops / t_gemm / 1e12 / fp8_peak, "work": "2 M N K FP8 (E5M2) MMA flops"}
    bound = "alu" if t_floor_alu >= t_floor_tensor else "tensor"
    main, other = (alu_view, tensor_view) if bound == "alu" else (tensor_view, alu_view)
    sh_ops = sum(l.M * l.N * (l.K // LLM_GROUP_S) * 4 for l in layers)
    t_sh_gemm = sum(gemm_sh) / 1e3
    return {"workload": "llama2_7b_block_linears", "tokens": layers[0].M,
            "layers": [f"{l.name}:{l.K}->{l.N}" for l in layers], "group_q": GROUP_Q,
            "group_s": LLM_GROUP_S, "code_bits": 16, "gemm": "tcgen05 (E5M2 operands)",
            "value": ops / t_tc / 1e12, "unit": "TOPS", "ms_per_step": t_tc * 1e3,
            "gemm_tops": ops / t_gemm / 1e12, "gemm_per_layer_ms": gemm_tc,
            "fused": {"value": ops / t_fused / 1e12, "unit": "TOPS", "ms_per_step": t_fused * 1e3,
                      "path": "quartz_linear_f16_ex per layer with prepared weights (16-bit codes "
                              "encoded straight into the E5M2 operand; bit-identical to quantize + linear)"},
            "roofline": dict(main, bound=bound, kernel="gemm_tcgen05_kernel",
                             **{("tensor" if bound == "alu" else "alu"): other},
                             floors_ms={"alu": t_floor_alu * 1e3, "tensor": t_floor_tensor * 1e3}),
            "shift": {"gemm": "accumulator-shift (exact 64-bit group sums)",
                      "tuning": "untuned: a plain 64 x 64-tile CUDA-core kernel (dp4a, shared-memory tiles), "
                                "kept as the exact reference schedule; its gap to the tuned tcgen05 GEMM is "
                                "not a like-for-like comparison",
                      "value": ops / t_sh / 1e12,
                      "ms_per_step": t_sh * 1e3, "gemm_per_layer_ms": gemm_sh,
                      "roofline": {"bound": "alu", "kernel": "gemm_shift_kernel",
                                   "achieved": sh_ops / t_sh_gemm / 1e12, "peak": alu_peak,
                                   "unit": "Top/s", "frac": sh_ops / t_sh_gemm / 1e12 / alu_peak,
                                   "work": "2 dp4a + 1 shift + 1 add per output per 8-wide subgroup"}},
            "peak_source": f"alu: {n_sm} SMs x {FP32_LANES_PER_SM} lanes x {sm_mhz:.0f} MHz ({peak_src} "
                           f"max SM clock); tensor: {fp8_src}",
            "encode": {"kernel": "quantize_sym_kernel<8, wide>", "per_layer_ms": quant_ms,
                       "gbs": enc_bytes / (sum(quant_ms) / 1e3) / 1e9},
            "inputs": "seeded synthetic Laplace(0,0.05), 0.2% channels x100; weights N(0,0.02)"}


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
