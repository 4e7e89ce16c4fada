"""PIFA layer forward throughput on GB300.

Default workload (one step = one pifa_forward over one token batch): the LLaMA-2-7B-shaped
attention projection m = n = 4096, r = 2048, decode batch T = 8 (bf16). The step runs the whole
hot path (selector, Y_p = X W_p^T, Y_np = Y_p C^T, both scatters into Y).

Printed as one JSON line on rank 0:
  value      tokens/s, device-timed (CUDA events on the launching stream) over K steps replayed
             from a CUDA graph; the weights rotate over enough copies that the working set is
             larger than L2 (every step streams its weights from HBM);
  e2e        the same metric through the public API with host buffers: per step, X copied from
             pinned host memory, pifa_forward, Y copied back to pinned host memory, in groups of
             four steps whose copies overlap the neighbouring groups' forwards (two copy streams,
             two groups in flight); the serial loop (no overlap) is reported beside it;
  roofline   the decode call's achieved HBM GB/s against MEASURED_PEAKS.json (algorithmic bytes:
             2 r(m + n - r) weight bytes + 2 T (n + m) activation bytes + 4 m index bytes);
  cpu_baseline  the fp64 oracle (numpy) on the host cores over a bounded sample of the workload;
  comparators   dense X W^T and low-rank (X V) U^T on the same GPU via torch.matmul;
  prefill    the same layer at T = 2048 (tcgen05 path) with its bf16 tensor roofline.

--impl reference times the oracle instead (the reference arm: the paper has no code).
Multi-GPU (torchrun): every rank runs an independent replica of the workload ("replicas only");
the time is the max over ranks and value sums the ranks' tokens.
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
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# BLAS threads of the oracle timings, fixed before numpy loads its BLAS: the host cores this
# process may run on, unless the caller chose (OpenBLAS reads its own variable first)
os.environ.setdefault("OPENBLAS_NUM_THREADS", str(len(os.sched_getaffinity(0))))
BLAS_THREADS = int(os.environ["OPENBLAS_NUM_THREADS"])

import numpy as np  # noqa: E402

from paper_2501_19090_gb300 import inputs  # noqa: E402

METRIC = "PIFA layer tokens/s at 1 GB300 + % of HBM / bf16 tensor roofline vs low-rank"
SHAPE = inputs.ATTN7B
T_DECODE = 8
T_PREFILL = 2048

# DRAM traffic per launch measured with ncu for a given kernel source (sha256 of the .cu file).
# A mismatch (the kernel changed since the capture) reports traffic as null.
NCU_TRAFFIC = {
    # decode_rows phase 1 + phase 2 of one call, attn 4096x4096 r=2048 T=8:
    # dram__bytes_read.sum 16.89 MB + 8.51 MB, dram__bytes_write.sum 0 (profiles/decode_attn7b_T8_ncu_full.md)
    "decode": {"sha": "fc56ea4f2ef87b8d", "bytes": 16885248 + 8512256},
}


def _src_sha(name: str) -> str:
    p = os.path.join(ROOT, "paper_2501_19090_gb300", "csrc", name)
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def decode_bytes(T, m, n, r):
    return 2 * r * (m + n - r) + 2 * T * (n + m) + 4 * m


def pifa_flops(T, m, n, r):
    return 2 * T * r * (m + n - r)


class ClockSampler:
    """nvidia-smi clocks, throttle reasons, memory clock and GPU / HBM temperatures sampled every
    100 ms while active (the state each timed region ran in)."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")
    EXTRA = ",clocks.mem,temperature.gpu,temperature.memory"
    _query = None  # Q + EXTRA where this nvidia-smi accepts the extra fields, else Q

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def _pick_query(self):
        if ClockSampler._query is None:
            ClockSampler._query = self.Q
            try:
                r = subprocess.run(["nvidia-smi", f"--query-gpu={self.Q + self.EXTRA}", "--format=csv,noheader,nounits",
                                    "-i", str(self.gpu)], capture_output=True, text=True, timeout=20)
                if r.returncode == 0 and len(r.stdout.strip().split(",")) >= 11:
                    ClockSampler._query = self.Q + self.EXTRA
            except Exception:
                pass
        return ClockSampler._query

    def __enter__(self):
        try:
            q = self._pick_query()
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", str(self.gpu)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        extra = {"mem_mhz": [], "gpu_temp_c": [], "hbm_temp_c": []}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
            for key, val in zip(("mem_mhz", "gpu_temp_c", "hbm_temp_c"), parts[8:11]):
                try:
                    extra[key].append(float(val))
                except ValueError:
                    pass
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        out = {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
               "samples": len(sm)}
        if extra["mem_mhz"]:
            out["mem_mhz"] = statistics.median(extra["mem_mhz"])
        for key in ("gpu_temp_c", "hbm_temp_c"):
            if extra[key]:
                out[key] = [min(extra[key]), max(extra[key])]
        return out


# ---------------------------------------------------------------------------------------------
def build_layer(shape, seed, c_dtype="bf16"):
    """Host-side setup: the library's compression (Algorithm 1); W_p rounded to bf16 and C to the
    chosen storage type (bf16 by default, or fp16)."""
    from paper_2501_19090_gb300 import pifa as P
    U, V, _ = inputs.make_factors(shape.m, shape.n, shape.r, seed)
    piv, nonp, Wp, C, info = P.pifa_compress(U, V, shape.r)
    Cq = inputs.round_fp16(C) if c_dtype == "fp16" else inputs.round_bf16(C)
    return dict(U=U, V=V, piv=piv, nonp=nonp, Wp=inputs.round_bf16(Wp), C=Cq, info=info, c_dtype=c_dtype)


# --shape: the decode measurement on another decode-config layer shape (profiling; the default line
# is the 7B attention layer). Other shapes use seeded random operands (inputs.synthetic_layer): the
# kernels' time does not depend on the values, and Algorithm 1 on a 28672 x 8192 layer takes minutes
# on the host.
SHAPES = {s.name: s for s in (inputs.ATTN7B, inputs.MLP7B_GATE, inputs.MLP7B_DOWN, inputs.ATTN70B,
                              inputs.MLP70B_GATE)}


def synthetic_layer_dict(shape, c_dtype="bf16"):
    piv, nonp, Wp, C = inputs.synthetic_layer(shape.m, shape.n, shape.r, 0)
    Cq = inputs.round_fp16(C) if c_dtype == "fp16" else C
    return dict(piv=piv.astype(np.int32), nonp=nonp.astype(np.int32), Wp=Wp, C=Cq, c_dtype=c_dtype)


def _torch_c_dtype(lay):
    import torch
    return torch.float16 if lay["c_dtype"] == "fp16" else torch.bfloat16


def _pifa_c_dtype(lay):
    from paper_2501_19090_gb300 import pifa as P
    return P.PIFA_DTYPE_FP16 if lay["c_dtype"] == "fp16" else P.PIFA_DTYPE_BF16


def run_ours(args, rank, world, local_rank):
    import torch
    from paper_2501_19090_gb300 import pifa as P

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    P.load()
    hbm_peak, tc_peak, tc_sust, peak_src = _peaks()
    shape = SHAPES[args.shape]
    m, n, r = shape.m, shape.n, shape.r
    T = args.tokens
    lay = (build_layer(shape, seed=0, c_dtype=args.c_dtype) if shape is SHAPE
           else synthetic_layer_dict(shape, args.c_dtype))
    bf = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev).to(torch.bfloat16)
    piv = torch.from_numpy(lay["piv"]).to(dev)
    nonp = torch.from_numpy(lay["nonp"]).to(dev)
    Wp0 = bf(lay["Wp"])
    C0 = torch.from_numpy(np.ascontiguousarray(lay["C"])).to(dev).to(_torch_c_dtype(lay))
    cdt = _pifa_c_dtype(lay)
    wbytes = (Wp0.numel() + C0.numel()) * 2
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    copies = max(4, math.ceil(3 * l2 / wbytes))
    Wps = [Wp0.clone() for _ in range(copies)]
    Cs = [C0.clone() for _ in range(copies)]
    rng = np.random.default_rng(1 + rank)
    Xs = [bf(inputs.make_activations(rng, T, n, "bf16")) for _ in range(copies)]
    Ys = [torch.empty((T, m), dtype=torch.bfloat16, device=dev) for _ in range(copies)]
    variant = P.pifa_select_variant(T, m, n, r, cdt)
    ws = P.workspace(P.pifa_workspace_size(T, m, n, r, variant, cdt), dev)
    stream = torch.cuda.Stream(device=dev)

    def step(i):
        j = i % copies
        P.pifa_forward(Xs[j], Wps[j], Cs[j], piv, nonp, Y=Ys[j], variant=variant, workspace_tensor=ws,
                       stream=stream)

    # warm-up (eager), then capture a graph of `per_graph` steps
    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            step(i)
    stream.synchronize()
    assert P.pifa_device_status(stream) == P.PIFA_OK
    per_graph = copies * max(1, 64 // copies)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(per_graph):
            step(i)
    replays = max(1, math.ceil(args.steps / per_graph))
    steps = replays * per_graph
    with torch.cuda.stream(stream):                # replays launch on the current stream
        for _ in range(max(3, args.warmup)):
            g.replay()
    stream.synchronize()

    dist = _dist()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clk:
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(replays):
                g.replay()
            e1.record(stream)
        torch.cuda.synchronize()
    if dist:
        dist.barrier()
    ms = e0.elapsed_time(e1)
    st = P.pifa_device_status(stream)
    assert st == P.PIFA_OK, P.pifa_status_string(st)
    ms_max = _max_over_ranks(ms)
    step_ms = ms_max / steps
    value = _job_value(world, T, steps, ms_max)
    achieved = decode_bytes(T, m, n, r) / (step_ms / 1e3) / 1e9

    # --- e2e through the public API with pinned host buffers ---
    Xh = torch.empty((T, n), dtype=torch.bfloat16).pin_memory()
    Xh.copy_(Xs[0].cpu())
    Yh = torch.empty((T, m), dtype=torch.bfloat16).pin_memory()
    Xd = torch.empty((T, n), dtype=torch.bfloat16, device=dev)
    e2e_steps = min(steps, 2000)
    with torch.cuda.stream(stream):
        for i in range(5):
            Xd.copy_(Xh, non_blocking=True)
            P.pifa_forward(Xd, Wps[i % copies], Cs[i % copies], piv, nonp, Y=Ys[0], variant=variant,
                                      workspace_tensor=ws, stream=stream)
            Yh.copy_(Ys[0], non_blocking=True)
    stream.synchronize()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for i in range(e2e_steps):
            Xd.copy_(Xh, non_blocking=True)
            P.pifa_forward(Xd, Wps[i % copies], Cs[i % copies], piv, nonp, Y=Ys[0], variant=variant,
                           workspace_tensor=ws, stream=stream)
            Yh.copy_(Ys[0], non_blocking=True)
        e1.record(stream)
    stream.synchronize()
    e2e_ms = _max_over_ranks(e0.elapsed_time(e1))
    e2e_eager = _job_value(world, T, e2e_steps, e2e_ms)
    # The same loop -- per step the upload of X from pinned host memory, pifa_forward, the download
    # of Y -- captured once as a CUDA graph and replayed, as a serving loop issues it: every step
    # still moves its bytes host -> device -> host; the graph removes the per-call host overhead.
    nh = 4
    Xhs = [torch.empty((T, n), dtype=torch.bfloat16).pin_memory() for _ in range(nh)]
    Yhs = [torch.empty((T, m), dtype=torch.bfloat16).pin_memory() for _ in range(nh)]
    for i in range(nh):
        Xhs[i].copy_(Xs[i % copies].cpu())
    per_e2e = copies * max(1, 64 // copies)

    def e2e_step(i):
        Xd.copy_(Xhs[i % nh], non_blocking=True)
        P.pifa_forward(Xd, Wps[i % copies], Cs[i % copies], piv, nonp, Y=Ys[0], variant=variant, workspace_tensor=ws,
                       stream=stream)
        Yhs[i % nh].copy_(Ys[0], non_blocking=True)

    ge = torch.cuda.CUDAGraph()
    with torch.cuda.graph(ge, stream=stream):
        for i in range(per_e2e):
            e2e_step(i)
    e2e_replays = max(1, e2e_steps // per_e2e)
    with torch.cuda.stream(stream):
        for _ in range(2):
            ge.replay()
    stream.synchronize()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(e2e_replays):
            ge.replay()
        e1.record(stream)
    stream.synchronize()
    e2e_graph = _job_value(world, T, e2e_replays * per_e2e, _max_over_ranks(e0.elapsed_time(e1)))
    assert np.array_equal(Yhs[(per_e2e - 1) % nh].float().numpy(), Ys[0].cpu().float().numpy())
    e2e_pipe, e2e_pipe_steps, e2e_pipe_per = e2e_pipelined(P, dev, T, n, m, Xhs, Wps, Cs, piv, nonp, variant, ws,
                                                           stream, world, e2e_steps)

    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{shape.name} {'decode' if T <= 16 else 'prefill'} T={T}", "m": m, "n": n, "r": r,
                   "tokens_per_step": T, "c_dtype": lay["c_dtype"],
                   "variant": P.pifa_variant_name(variant), "parallelism": f"replicas{world}",
                   "l2_defeat": f"{copies} rotating weight copies ({copies * wbytes / 1e6:.0f} MB > 3x L2)",
                   "timing": "CUDA graph replay, CUDA events on the launching stream"},
        "e2e": {"value": e2e_pipe, "unit": "tokens/s", "h2d_bytes_per_step": T * n * 2,
                "d2h_bytes_per_step": T * m * 2,
                "mode": f"serving loop: per step X uploaded from pinned host memory (one copy per step), "
                        f"pifa_forward, Y downloaded to pinned host memory (one copy per step); steps in groups of "
                        f"4 with two groups in flight, uploads and downloads on two copy streams overlapping the "
                        f"neighbouring groups' forwards, the compute stream waiting on the copies once per group; "
                        f"{e2e_pipe_per} steps per CUDA graph, {e2e_pipe_steps} steps timed; the last step's Y "
                        f"checked against a separate forward",
                "serial_value": e2e_eager,
                "serial_mode": "the same steps one after another on one stream, issued call by call (no overlap)",
                "serial_graph_value": e2e_graph,
                "serial_graph_mode": "the serial loop captured as a CUDA graph and replayed"},
        "roofline": ({"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                      "frac": achieved / hbm_peak,
                      "traffic": _traffic("decode.cu", "decode") if (T, m, n, r) == (8, 4096, 4096, 2048) else None,
                      "peak_source": f"{peak_src} hbm_gbs",
                      "kernel": "decode phase 1 + phase 2 (one PDL-chained pair per call)",
                      "algorithmic_bytes_per_launch": decode_bytes(T, m, n, r)} if T <= 16 else
                     {"bound": "tensor", "achieved": pifa_flops(T, m, n, r) / (step_ms / 1e3) / 1e12, "peak": tc_peak,
                      "unit": "TFLOP/s", "frac": pifa_flops(T, m, n, r) / (step_ms / 1e3) / 1e12 / tc_peak,
                      "traffic": None, "peak_source": f"{peak_src} bf16_tflops (burst)",
                      "kernel": f"{P.pifa_variant_name(variant)} prefill (GEMM 1 + GEMM 2 per call)",
                      "algorithmic_flops_per_launch": pifa_flops(T, m, n, r)}),
        "gpu_launches": steps * (2 if m > r else 1),
        "clocks": clk.summary(),
    }
    if rank == 0 and world == 1 and not args.no_extras and shape is SHAPE:
        # one GPU only (at N > 1 every GPU would wait for rank 0's extras); the HBM-bound points first: the prefill-sized GEMMs after them hold the power cap
        with ClockSampler(local_rank) as clk_x:
            out["decode_sweep"] = decode_sweep(dev, stream, hbm_peak, peak_src)
            out["grouped_mlp7b_gate_up"] = grouped_point(dev, stream, hbm_peak, tc_peak, peak_src)
        out["decode_sweep_clocks"] = clk_x.summary()
        with ClockSampler(local_rank) as clk_p:
            out["comparators"] = comparators(dev, lay, T, copies, stream)
            out["prefill"] = prefill_point(dev, lay, copies, stream, tc_peak, peak_src)
            out["prefill_fused"] = prefill_point(dev, lay, copies, stream, tc_peak, peak_src,
                                                 variant=P.PIFA_VARIANT_PREFILL_FUSED)
        out["prefill_clocks"] = clk_p.summary()
        out["cpu_baseline"] = cpu_baseline(lay, T)
    return out


def comparators(dev, lay, T, copies, stream):
    """Dense X W^T and two-factor low-rank (X V) U^T on the same GPU (torch.matmul, bf16), each a
    CUDA graph over rotating weight copies timed in steady state (_graph_ms)."""
    import torch
    res = {}
    U = torch.from_numpy(lay["U"]).to(dev).to(torch.bfloat16)
    V = torch.from_numpy(lay["V"]).to(dev).to(torch.bfloat16)
    W = (U.float() @ V.float().t()).to(torch.bfloat16)
    for Tq in (T, T_PREFILL):
        X = torch.randn((Tq, V.shape[0]), device=dev).to(torch.bfloat16)
        Ws = [W.clone() for _ in range(max(2, copies // 2))]
        Us = [U.clone() for _ in range(copies)]
        Vs = [V.clone() for _ in range(copies)]
        for name, fn, nrot in (("dense", lambda i: X @ Ws[i % len(Ws)].t(), len(Ws)),
                               ("lowrank", lambda i: (X @ Vs[i % copies]) @ Us[i % copies].t(), copies)):
            with torch.cuda.stream(stream):
                for i in range(5):
                    fn(i)
            stream.synchronize()
            per = nrot * max(1, 64 // nrot) if Tq <= 16 else nrot
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i in range(per):
                    fn(i)
            ms = _graph_ms(g, stream) / per
            del g
            res[f"{name}_T{Tq}"] = {"tokens_per_s": Tq / (ms / 1e3), "ms": ms}
    return res


DECODE_SWEEP = [(inputs.ATTN7B, (1, 8, 16)), (inputs.MLP7B_GATE, (1, 8)), (inputs.MLP7B_DOWN, (1, 8)),
                (inputs.ATTN70B, (1, 8, 16)), (inputs.MLP70B_GATE, (1, 8, 16))]


def decode_sweep(dev, stream, hbm_peak, peak_src):
    """The decode variant on every decode-sized layer shape (HBM-bound), beside the two-factor
    low-rank layer of the same shape. Timing inputs only: W_p and C are seeded N(0, 1) bf16 and the
    pivot set a seeded random r-subset (kernel time does not depend on the values); weight copies
    rotate so that every call streams its weights from HBM."""
    import torch
    from paper_2501_19090_gb300 import pifa as P
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    out = []
    for shape, Ts in DECODE_SWEEP:
        m, n, r = shape.m, shape.n, shape.r
        rng = np.random.default_rng(11)
        perm = rng.permutation(m)
        piv = torch.from_numpy(np.sort(perm[:r]).astype(np.int32)).to(dev)
        nonp = torch.from_numpy(np.sort(perm[r:]).astype(np.int32)).to(dev)
        gen = torch.Generator(device=dev)
        gen.manual_seed(12)
        wbytes = 2 * r * (m + n - r)
        copies = max(4, math.ceil(3 * l2 / wbytes))  # as the main line: every call streams from HBM
        Wps = [torch.randn((r, n), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
        Cs = [torch.randn((m - r, r), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
        lr_copies = max(4, math.ceil(3 * l2 / (2 * r * (m + n))))
        Us = [torch.randn((m, r), device=dev, generator=gen).to(torch.bfloat16) for _ in range(lr_copies)]
        Vs = [torch.randn((n, r), device=dev, generator=gen).to(torch.bfloat16) for _ in range(lr_copies)]
        for T in Ts:
            # per weight copy its own X and Y, as the main line
            Xc = [torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
            Yc = [torch.empty((T, m), dtype=torch.bfloat16, device=dev) for _ in range(copies)]
            X = Xc[0]
            variant = P.pifa_select_variant(T, m, n, r, P.PIFA_DTYPE_BF16)
            ws = P.workspace(P.pifa_workspace_size(T, m, n, r, variant), dev, tag="sweep")

            def step(i):
                j = i % copies
                P.pifa_forward(Xc[j], Wps[j], Cs[j], piv, nonp, Y=Yc[j], variant=variant,
                               workspace_tensor=ws, stream=stream)

            with torch.cuda.stream(stream):
                for i in range(4):
                    step(i)
            per_graph = copies * max(1, 64 // copies)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i in range(per_graph):
                    step(i)
            ms = _graph_ms(g, stream, replays=max(3, 256 // per_graph)) / per_graph
            assert P.pifa_device_status(stream) == P.PIFA_OK
            lr = lambda i: (X @ Vs[i % lr_copies]) @ Us[i % lr_copies].t()
            with torch.cuda.stream(stream):
                for i in range(4):
                    lr(i)
            g2 = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g2, stream=stream):
                for i in range(per_graph):
                    lr(i)
            lr_ms = _graph_ms(g2, stream, replays=max(3, 256 // per_graph)) / per_graph
            gbs = decode_bytes(T, m, n, r) / (ms / 1e3) / 1e9
            out.append({"workload": f"{shape.name} decode T={T}", "us_per_call": ms * 1e3,
                        "tokens_per_s": T / (ms / 1e3), "hbm_gbs": gbs, "frac": gbs / hbm_peak,
                        "lowrank_us_per_call": lr_ms * 1e3, "speedup_vs_lowrank": lr_ms / ms,
                        "weight_copies": copies, "peak_source": f"{peak_src} hbm_gbs"})
            del g, g2
        del Wps, Cs, Us, Vs
        torch.cuda.empty_cache()
    return out


def grouped_point(dev, stream, hbm_peak, tc_peak, peak_src):
    """The 7B MLP's gate and up projections (11008 x 4096, r = 2048) sharing X: one
    pifa_forward_grouped call against two pifa_forward calls, graph replay, >= 4 rotating weight
    copies; timing operands as in decode_sweep (seeded N(0, 1) weights, random pivot sets)."""
    import torch
    from paper_2501_19090_gb300 import pifa as P
    shape = inputs.MLP7B_GATE
    m, n, r, G = shape.m, shape.n, shape.r, 2
    rng = np.random.default_rng(13)
    piv_l, nonp_l = [], []
    for g in range(G):
        perm = rng.permutation(m)
        piv_l.append(torch.from_numpy(np.sort(perm[:r]).astype(np.int32)).to(dev))
        nonp_l.append(torch.from_numpy(np.sort(perm[r:]).astype(np.int32)).to(dev))
    piv_s = torch.cat([piv_l[g] + g * m for g in range(G)])
    nonp_s = torch.cat([nonp_l[g] + g * m for g in range(G)])
    gen = torch.Generator(device=dev)
    gen.manual_seed(14)
    copies = 4
    Wps = [torch.randn((G * r, n), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
    Cs = [torch.randn((G * (m - r), r), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
    out = []
    for T in (1, 8, T_PREFILL):
        X = torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16)
        Y = torch.empty((T, G * m), dtype=torch.bfloat16, device=dev)
        Ys = [torch.empty((T, m), dtype=torch.bfloat16, device=dev) for _ in range(G)]
        ws1 = P.workspace(P.pifa_workspace_size(T, m, n, r), dev, tag="grp1")
        wsg = P.workspace(P.pifa_workspace_size_grouped(G, T, m, n, r), dev, tag="grpG")

        def sep(i):
            j = i % copies
            for g in range(G):
                P.pifa_forward(X, Wps[j][g * r:(g + 1) * r], Cs[j][g * (m - r):(g + 1) * (m - r)], piv_l[g],
                               nonp_l[g], Y=Ys[g], workspace_tensor=ws1, stream=stream)

        def grp(i):
            j = i % copies
            P.pifa_forward_grouped(G, X, Wps[j], Cs[j], piv_s, nonp_s, Y=Y, workspace_tensor=wsg, stream=stream)

        per_graph = 16 if T <= 16 else 4
        res = {}
        for name, fn in (("separate", sep), ("grouped", grp)):
            with torch.cuda.stream(stream):
                for i in range(4):
                    fn(i)
            g_ = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_, stream=stream):
                for i in range(per_graph):
                    fn(i)
            res[name] = _graph_ms(g_, stream, replays=5) / per_graph
            del g_
        assert P.pifa_device_status(stream) == P.PIFA_OK
        e = {"workload": f"{shape.name} x2 (gate + up) T={T}", "grouped_us": res["grouped"] * 1e3,
             "separate_us": res["separate"] * 1e3, "speedup": res["separate"] / res["grouped"]}
        if T <= 16:
            gbs = G * decode_bytes(T, m, n, r) / res["grouped"] / 1e6
            e.update({"hbm_gbs": gbs, "frac": gbs / hbm_peak, "peak_source": f"{peak_src} hbm_gbs"})
        else:
            tf = G * pifa_flops(T, m, n, r) / res["grouped"] / 1e9
            e.update({"tflops": tf, "frac": tf / tc_peak, "peak_source": f"{peak_src} bf16_tflops (burst)"})
        out.append(e)
    del Wps, Cs
    torch.cuda.empty_cache()
    return out


def e2e_pipelined(P, dev, T, n, m, Xhs, Wps, Cs, piv, nonp, variant, ws, stream, world, steps):
    """End to end through pifa_forward as a serving loop issues it: every step uploads its own X
    from pinned host memory, runs its forward and downloads its own Y to pinned host memory. Steps
    go in groups of K: a group's K uploads (one copy per step) on an upload stream, its K forwards
    back to back on the compute stream, its K downloads (one copy per step) on a download stream,
    with two groups' buffers in flight so that one group's copies overlap the neighbouring groups'
    forwards. The compute stream waits on the copies once per group, so that the forwards of a
    group follow one another with programmatic dependent launch, as in the device-only line (a
    wait before every forward measured 15.5 µs per step at T = 8 against 8.8 µs of kernel time).
    Captured as one multi-stream CUDA graph of `per` steps and replayed; a replay starts after the
    previous one has drained, so each replay pays one pipeline fill. Returns (tokens/s over all
    ranks, steps timed, per)."""
    import torch
    K, NG = 4, 2                                   # steps per group, groups in flight
    nh = len(Xhs)
    copies = len(Wps)
    Xd = [torch.empty((T, n), dtype=torch.bfloat16, device=dev) for _ in range(K * NG)]
    Yd = [torch.empty((T, m), dtype=torch.bfloat16, device=dev) for _ in range(K * NG)]
    Yhs = [torch.empty((T, m), dtype=torch.bfloat16).pin_memory() for _ in range(nh)]
    s_in = torch.cuda.Stream(device=dev)
    s_out = torch.cuda.Stream(device=dev)
    per = K * math.ceil(copies * max(1, 64 // copies) / K)

    def pipeline(k_steps):
        ev_in = [torch.cuda.Event() for _ in range(NG)]
        ev_fwd = [torch.cuda.Event() for _ in range(NG)]
        ev_out = [torch.cuda.Event() for _ in range(NG)]
        fork = torch.cuda.Event()
        fork.record(stream)
        s_in.wait_event(fork)
        s_out.wait_event(fork)
        for j in range(k_steps // K):
            gb = j % NG                            # the group's buffer set
            if j >= NG:
                s_in.wait_event(ev_fwd[gb])        # group j - NG's forwards have read Xd
            with torch.cuda.stream(s_in):
                for t in range(K):
                    i = j * K + t
                    Xd[gb * K + t].copy_(Xhs[i % nh], non_blocking=True)
            ev_in[gb].record(s_in)
            stream.wait_event(ev_in[gb])
            if j >= NG:
                stream.wait_event(ev_out[gb])      # group j - NG's downloads have read Yd
            for t in range(K):
                i = j * K + t
                P.pifa_forward(Xd[gb * K + t], Wps[i % copies], Cs[i % copies], piv, nonp, Y=Yd[gb * K + t],
                               variant=variant, workspace_tensor=ws, stream=stream)
            ev_fwd[gb].record(stream)
            s_out.wait_event(ev_fwd[gb])
            with torch.cuda.stream(s_out):
                for t in range(K):
                    i = j * K + t
                    Yhs[i % nh].copy_(Yd[gb * K + t], non_blocking=True)
            ev_out[gb].record(s_out)
        join_in, join_out = torch.cuda.Event(), torch.cuda.Event()
        join_in.record(s_in)
        join_out.record(s_out)
        stream.wait_event(join_in)
        stream.wait_event(join_out)

    with torch.cuda.stream(stream):
        pipeline(2 * K * NG)                       # eager warm-up of the same streams and buffers
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        pipeline(per)
    replays = max(1, steps // per)
    with torch.cuda.stream(stream):
        for _ in range(2):
            g.replay()
    stream.synchronize()
    dist = _dist()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(replays):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    ms = _max_over_ranks(e0.elapsed_time(e1))
    # the last step's downloaded Y equals a separate forward of the same inputs (decode and prefill
    # are deterministic)
    i = per - 1
    with torch.cuda.stream(stream):
        Xchk = Xhs[i % nh].to(dev)
        Ychk = torch.empty((T, m), dtype=torch.bfloat16, device=dev)
        P.pifa_forward(Xchk, Wps[i % copies], Cs[i % copies], piv, nonp, Y=Ychk, variant=variant,
                       workspace_tensor=ws, stream=stream)
    stream.synchronize()
    assert torch.equal(Yhs[i % nh].view(torch.int16), Ychk.cpu().view(torch.int16)), "pipelined e2e output mismatch"
    return _job_value(world, T, replays * per, ms), replays * per, per


def _graph_ms(g, stream, replays=None, warm_s=0.1, timed_s=0.25):
    """Milliseconds per replay of graph g, every replay on `stream`: about warm_s seconds of
    replays first, then at least `replays` (or about timed_s seconds of) replays timed with events
    on the same stream. (CUDAGraph.replay() launches on the current stream; a warm-up replayed on
    the default stream is not waited for by a side stream's start event, and its tail would be
    timed as well.)"""
    import torch
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        g.replay()
        e1.record(stream)
        stream.synchronize()
        one = max(e0.elapsed_time(e1) / 1e3, 1e-6)       # seconds per replay, first estimate
        for _ in range(max(2, math.ceil(warm_s / one))):
            g.replay()
        stream.synchronize()
        n_rep = max(replays or 3, math.ceil(timed_s / one))
        e0.record(stream)
        for _ in range(n_rep):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / n_rep


def _eager_ms(call, stream, warm_s=0.1, timed_s=0.25):
    """Milliseconds per call(i) issued eagerly on `stream` (calls long enough that the host keeps
    ahead), in steady state as _graph_ms: about warm_s seconds of calls first, then about timed_s
    seconds timed."""
    import torch
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for i in range(4):
            call(i)
        e1.record(stream)
    stream.synchronize()
    one = max(e0.elapsed_time(e1) / 4e3, 1e-6)
    with torch.cuda.stream(stream):
        for i in range(math.ceil(warm_s / one)):
            call(i)
        n_call = max(8, math.ceil(timed_s / one))
        e0.record(stream)
        for i in range(n_call):
            call(i)
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / n_call


def prefill_point(dev, lay, copies, stream, tc_peak, peak_src, variant=None):
    import torch
    from paper_2501_19090_gb300 import pifa as P
    m, n, r = SHAPE.m, SHAPE.n, SHAPE.r
    T = T_PREFILL
    bf = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev).to(torch.bfloat16)
    piv = torch.from_numpy(lay["piv"]).to(dev)
    nonp = torch.from_numpy(lay["nonp"]).to(dev)
    Wp = bf(lay["Wp"])
    C = torch.from_numpy(np.ascontiguousarray(lay["C"])).to(dev).to(_torch_c_dtype(lay))
    cdt = _pifa_c_dtype(lay)
    ncp = max(2, copies // 4)
    Wps = [Wp.clone() for _ in range(ncp)]
    Cs = [C.clone() for _ in range(ncp)]
    rng = np.random.default_rng(5)
    Xs = [bf(inputs.make_activations(rng, T, n, "bf16")) for _ in range(ncp)]
    Y = torch.empty((T, m), dtype=torch.bfloat16, device=dev)
    if variant is None:
        variant = P.pifa_select_variant(T, m, n, r, cdt)
    ws = P.workspace(P.pifa_workspace_size(T, m, n, r, variant, cdt), dev, tag="prefill")
    with torch.cuda.stream(stream):
        for i in range(5):
            P.pifa_forward(Xs[i % ncp], Wps[i % ncp], Cs[i % ncp], piv, nonp, Y=Y, variant=variant,
                           workspace_tensor=ws, stream=stream)
    stream.synchronize()

    def call(i):
        P.pifa_forward(Xs[i % ncp], Wps[i % ncp], Cs[i % ncp], piv, nonp, Y=Y, variant=variant,
                       workspace_tensor=ws, stream=stream)

    ms = _eager_ms(call, stream)
    assert P.pifa_device_status(stream) == P.PIFA_OK
    tf = pifa_flops(T, m, n, r) / (ms / 1e3) / 1e12
    return {"workload": f"{SHAPE.name} prefill T={T}", "variant": P.pifa_variant_name(variant),
            "tokens_per_s": T / (ms / 1e3), "ms_per_step": ms,
            "roofline": {"bound": "tensor", "achieved": tf, "peak": tc_peak, "unit": "TFLOP/s",
                         "frac": tf / tc_peak, "peak_source": f"{peak_src} bf16_tflops (burst)",
                         "algorithmic_flops_per_launch": pifa_flops(T, m, n, r)}}


def cpu_baseline(lay, T, budget_s=10.0, single_s=5.0):
    """The fp64 oracle forward (numpy) on the host cores over a bounded sample of the workload,
    with BLAS_THREADS BLAS threads; the same forward on one thread, timed in a fresh interpreter
    (numpy's thread count is fixed when it loads), is reported beside it."""
    import oracle
    rng = np.random.default_rng(9)
    X = inputs.make_activations(rng, T, SHAPE.n, "bf16")
    Wp, C = lay["Wp"].astype(np.float64), lay["C"].astype(np.float64)
    piv, nonp = lay["piv"].astype(np.int64), lay["nonp"].astype(np.int64)
    oracle.forward(X, Wp, C, piv, nonp)
    t0 = time.perf_counter()
    calls = 0
    while time.perf_counter() - t0 < budget_s:
        oracle.forward(X, Wp, C, piv, nonp)
        calls += 1
    dt = time.perf_counter() - t0
    out = {"value": calls * T / dt, "unit": "tokens/s", "cores": BLAS_THREADS, "kind": "oracle",
           "sample": f"{calls} oracle forwards of T={T} tokens on {SHAPE.name} (fp64 numpy, "
                     f"{BLAS_THREADS} BLAS threads), {dt:.1f} s"}
    try:
        out["single_thread"] = _oracle_rate_one_thread(X, Wp, C, piv, nonp, T, single_s)
    except Exception as e:  # reported, never fatal: the main figure stands on its own
        out["single_thread"] = {"error": f"{type(e).__name__}: {e}"}
    return out


_ONE_THREAD_TIMER = """
import json, sys, time
import numpy as np
sys.path.insert(0, sys.argv[1])
import oracle
d = np.load(sys.argv[2])
args = (d["X"], d["Wp"], d["C"], d["piv"], d["nonp"])
oracle.forward(*args)
t0, calls = time.perf_counter(), 0
while time.perf_counter() - t0 < float(sys.argv[3]):
    oracle.forward(*args)
    calls += 1
print(json.dumps({"calls": calls, "seconds": time.perf_counter() - t0}))
"""


def _oracle_rate_one_thread(X, Wp, C, piv, nonp, T, budget_s):
    """Tokens/s of the oracle forward with one BLAS thread, in a fresh interpreter."""
    import tempfile
    with tempfile.TemporaryDirectory() as d:
        path = os.path.join(d, "case.npz")
        np.savez(path, X=X, Wp=Wp, C=C, piv=piv, nonp=nonp)
        env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
        r = subprocess.run([sys.executable, "-c", _ONE_THREAD_TIMER, ROOT, path, str(budget_s)], env=env,
                           capture_output=True, text=True, timeout=budget_s + 120)
    if r.returncode != 0:
        raise RuntimeError(r.stderr.strip().splitlines()[-1] if r.stderr.strip() else f"exit {r.returncode}")
    res = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": res["calls"] * T / res["seconds"], "unit": "tokens/s", "cores": 1,
            "sample": f"{res['calls']} oracle forwards, {res['seconds']:.1f} s, one BLAS thread"}


def _traffic(src, key):
    t = NCU_TRAFFIC.get(key)
    if not t or t.get("sha") != _src_sha(src):
        return None
    return t["bytes"]


# ---------------------------------------------------------------------------------------------
_DIST = None


def _dist():
    return _DIST


def _max_over_ranks(v):
    """The slowest rank's value (every rank gets it); a no-op on one process."""
    d = _dist()
    if not d:
        return v
    import torch
    dev = "cuda" if d.get_backend() == "nccl" else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    d.all_reduce(t, op=d.ReduceOp.MAX)
    return float(t.item())


def _job_value(world, tokens_per_step, steps, ms_max):
    """Whole-job tokens/s: each of `world` replicas ran `steps` steps of `tokens_per_step` tokens,
    and the job took as long as its slowest rank (`ms_max`)."""
    return world * tokens_per_step * steps / (ms_max / 1e3)


def run_reference(args, rank):
    """Reference arm: the fp64 oracle (the paper publishes no code) on the host cores, same workload."""
    import oracle
    from paper_2501_19090_gb300 import pifa as P
    if rank != 0:
        return None
    T = args.tokens
    U, V, _ = inputs.make_factors(SHAPE.m, SHAPE.n, SHAPE.r, 0)
    L = oracle.compress(U, V, SHAPE.r, "lapack")
    Cq = inputs.round_fp16(L.C) if args.c_dtype == "fp16" else inputs.round_bf16(L.C)
    Wp, C = inputs.round_bf16(L.Wp).astype(np.float64), Cq.astype(np.float64)
    rng = np.random.default_rng(1)
    X = inputs.make_activations(rng, T, SHAPE.n, "bf16")
    for _ in range(max(3, args.warmup)):
        oracle.forward(X, Wp, C, L.pivots, L.nonpivots)
    # bounded sample: at most ~60 s of oracle forwards, however many steps were asked for
    t0 = time.perf_counter()
    done = 0
    while done < args.steps and (done == 0 or time.perf_counter() - t0 < 60.0):
        oracle.forward(X, Wp, C, L.pivots, L.nonpivots)
        done += 1
    dt = time.perf_counter() - t0
    v = T * done / dt
    cores = BLAS_THREADS
    del P
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": done, "requested_steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / done,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": f"{SHAPE.name} decode T={T}", "m": SHAPE.m, "n": SHAPE.n,
                                            "r": SHAPE.r, "tokens_per_step": T},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{done} of {args.steps} requested fp64 oracle forwards of T={T} "
                                       f"(numpy, {cores} BLAS threads; capped at ~60 s)"},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    global _DIST
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--tokens", type=int, default=T_DECODE)
    ap.add_argument("--no-extras", action="store_true")
    ap.add_argument("--c-dtype", default="bf16", choices=["bf16", "fp16"])
    ap.add_argument("--shape", default=SHAPE.name, choices=sorted(SHAPES),
                    help="decode layer shape of the main line (other shapes: synthetic operands, no extras)")
    args = ap.parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        out = run_reference(args, rank)
        if out is not None:
            print(json.dumps(out), flush=True)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
        _DIST = dist
    out = run_ours(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if _DIST:
        _DIST.barrier()
        _DIST.destroy_process_group()


if __name__ == "__main__":
    main()
