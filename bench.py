"""PIFA layer forward throughput on GB300.

Headline workload (one step = one pifa_forward over one token batch): the LLaMA-2-70B-shaped MLP
gate/up projection m = 28672, n = 8192, r = 4096 (the largest layer of the workloads, one layer on
one GPU), decode batch T = 16, bf16. The step runs the whole hot path: the selector, Y_p = X W_p^T,
Y_np = Y_p C^T and both scatters into Y.

Printed as one JSON line on rank 0:
  value      tokens/s, device-timed with CUDA events on the launching stream over exactly --steps
             steps replayed from CUDA graphs; the timed region is repeated until the clock sampler
             has seen it (value = the median repetition); the weights rotate over enough copies
             that the working set exceeds L2, so every step streams its weights from HBM;
  e2e        the same metric through the public API with host buffers: per step X copied from
             pinned host memory, pifa_forward, Y copied back to pinned host memory (groups of four
             steps whose copies overlap the neighbouring groups' forwards); the serial loop beside it;
  roofline   achieved HBM GB/s of the call against MEASURED_PEAKS.json (algorithmic bytes
             2 r(m + n - r) + 2 T (n + m) + 4 m per call);
  comparators  the same shape as a dense layer (X W^T) and a two-factor low-rank layer
             ((X V) U^T) through torch.matmul on the same GPU, timed the same way;
  cpu_baseline the fp64 oracle (numpy) on the host cores over a bounded sample of the workload.
Extras (one GPU only): every decode configuration beside its low-rank and dense layers, the 7B MLP
as three layers back to back, the prefill configurations (7B attention T = 2048 / 8192, 70B q/o and
gate/up T = 4096) and the rank-fraction sweep at T = 2048, each with its roofline and clock record.

--impl reference times the oracle instead (the reference arm: the paper publishes no code).
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
SHAPE = inputs.MLP70B_GATE       # the headline layer
T_DECODE = 16

# DRAM traffic per call (dram__bytes_read.sum + dram__bytes_write.sum over the call's kernels)
# measured with ncu, keyed by (layer, T), with the sha256 prefixes of the kernel sources it was
# taken on. A source mismatch (a kernel changed since the capture) reports traffic as null.
NCU_TRAFFIC = {
    # profiles/decode_tc_gateup70b_T16_traffic.md: phase 1 in clusters of 8 CTAs per row block,
    # phase 2 one CTA per row block; two kernels, no partial sums in global memory
    ("llama2_70b_gate_up_28672x8192_r4096", 16): {
        "sha": {"decode_tc.cu": "35b8964778d8fafd", "decode.cu": "d641f7870ae488ab"},
        "bytes": 269409536,
    },
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


def lowrank_bytes(T, m, n, r):
    return 2 * r * (m + n) + 2 * T * (n + m)


def dense_bytes(T, m, n):
    return 2 * m * n + 2 * T * (n + m)


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
SHAPES = {s.name: s for s in (inputs.ATTN7B, inputs.MLP7B_GATE, inputs.MLP7B_DOWN, inputs.ATTN70B,
                              inputs.MLP70B_GATE)}


def timing_layer(shape, dev, seed, c_dtype="bf16", copies=1):
    """Device operands of one layer shape for timing: a seeded random ascending pivot set and its
    complement, W_p ~ N(0, 1/r) and C ~ N(0, 0.18^2) drawn on the GPU (bf16; C in c_dtype), in
    `copies` independent copies. The kernels' time does not depend on the values (the parity tests
    run the real compressed layers)."""
    import torch
    m, n, r = shape.m, shape.n, shape.r
    rng = np.random.default_rng(20_000 + seed)
    perm = rng.permutation(m)
    piv = torch.from_numpy(np.sort(perm[:r]).astype(np.int32)).to(dev)
    nonp = torch.from_numpy(np.sort(perm[r:]).astype(np.int32)).to(dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 + seed)
    cdt = torch.float16 if c_dtype == "fp16" else torch.bfloat16
    Wps = [_padded((torch.randn((r, n), device=dev, generator=gen) / math.sqrt(r)).to(torch.bfloat16))
           for _ in range(copies)]
    Cs = [_padded((torch.randn((m - r, r), device=dev, generator=gen) * 0.18).to(cdt)) for _ in range(copies)]
    return piv, nonp, Wps, Cs


def _padded(a):
    """a (rows x cols) copied into a buffer whose row pitch is cols rounded up to 8 elements (the
    library's 16-byte row rule); returns the rows x cols view."""
    import torch
    rows, cols = a.shape
    ld = (cols + 7) // 8 * 8
    if ld == cols:
        return a
    buf = torch.zeros((rows, ld), dtype=a.dtype, device=a.device)
    buf[:, :cols] = a
    return buf[:, :cols]


def _copies_for(dev, weight_bytes, lo=4):
    """Weight copies whose total exceeds 3x L2, so that a rotation streams every step from HBM."""
    import torch
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    return max(lo, math.ceil(3 * l2 / weight_bytes))


def _graph_of(fn, n, stream):
    """A CUDA graph of fn(0) .. fn(n - 1) captured on `stream` (after 3 eager warm-up calls)."""
    import torch
    with torch.cuda.stream(stream):
        for i in range(3):
            fn(i)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n):
            fn(i)
    return g


def _steady_us(fn, per_graph, stream):
    """Microseconds per fn call in steady state: a graph of per_graph calls, replayed on `stream`
    for ~0.1 s untimed then >= 0.25 s timed (_graph_ms)."""
    g = _graph_of(fn, per_graph, stream)
    us = _graph_ms(g, stream) / per_graph * 1e3
    del g
    return us


def _comparator_fns(dev, shape, T, gen, n_lr, n_dense):
    """Two-factor low-rank (X V) U^T and dense X W^T layers of the shape (bf16, torch.matmul on the
    same GPU), each over rotating weight copies: returns (lowrank fn, dense fn, X)."""
    import torch
    m, n, r = shape.m, shape.n, shape.r
    X = torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16)
    Us = [(torch.randn((m, r), device=dev, generator=gen) / math.sqrt(r)).to(torch.bfloat16) for _ in range(n_lr)]
    Vs = [(torch.randn((n, r), device=dev, generator=gen) / math.sqrt(r)).to(torch.bfloat16) for _ in range(n_lr)]
    Ws = [torch.randn((m, n), device=dev, generator=gen).to(torch.bfloat16) for _ in range(n_dense)]
    lr = lambda i: (X @ Vs[i % n_lr]) @ Us[i % n_lr].t()
    dense = lambda i: X @ Ws[i % n_dense].t()
    return lr, dense, X


def layer_point(dev, stream, shape, T, hbm_peak, tc_peak, peak_src, name=None, c_dtype="bf16"):
    """One layer shape at T tokens: the selected PIFA variant, the two-factor low-rank layer and the
    dense layer on the same GPU, each a CUDA graph replayed in steady state over rotating weight
    copies (decode: every copy's bytes exceed 3x L2 in total; prefill: two copies), with the
    roofline of the PIFA call (HBM for the decode variant, bf16 tensor otherwise) and the clocks seen."""
    import torch
    from paper_2501_19090_gb300 import pifa as P
    m, n, r = shape.m, shape.n, shape.r
    decode = is_decode(T, m, r)
    copies = _copies_for(dev, 2 * r * (m + n - r)) if decode else 2
    piv, nonp, Wps, Cs = timing_layer(shape, dev, 7, c_dtype, copies)
    gen = torch.Generator(device=dev)
    gen.manual_seed(17)
    Xs = [torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
    Ys = [torch.empty((T, m), dtype=torch.bfloat16, device=dev) for _ in range(copies)]
    cdt = P.PIFA_DTYPE_FP16 if c_dtype == "fp16" else P.PIFA_DTYPE_BF16
    variant = P.pifa_select_variant(T, m, n, r, cdt)
    ws = P.workspace(P.pifa_workspace_size(T, m, n, r, variant, cdt), dev, tag="point")

    def step(i):
        j = i % copies
        P.pifa_forward(Xs[j], Wps[j], Cs[j], piv, nonp, Y=Ys[j], variant=variant, workspace_tensor=ws, stream=stream)

    per = copies * max(1, 64 // copies) if decode else 8
    n_lr = _copies_for(dev, 2 * r * (m + n)) if decode else 2
    n_dense = _copies_for(dev, 2 * m * n, lo=2) if decode else 2
    with ClockSampler(torch.cuda.current_device()) as clk:
        us = _steady_us(step, per, stream)
        st = P.pifa_device_status(stream)
        assert st == P.PIFA_OK, P.pifa_status_string(st)
        del Wps, Cs, Xs, Ys
        torch.cuda.empty_cache()
        lr, dense, _ = _comparator_fns(dev, shape, T, gen, n_lr, n_dense)
        lr_us = _steady_us(lr, n_lr * max(1, 64 // n_lr) if decode else 8, stream)
        dense_us = _steady_us(dense, n_dense * max(1, 64 // n_dense) if decode else 8, stream)
    del lr, dense
    torch.cuda.empty_cache()
    out = {"workload": name or f"{shape.name} {'decode' if decode else 'prefill'} T={T}", "m": m, "n": n, "r": r,
           "T": T, "variant": P.pifa_variant_name(variant), "c_dtype": c_dtype, "us_per_call": us,
           "tokens_per_s": T / (us / 1e6), "lowrank_us": lr_us, "dense_us": dense_us,
           "speedup_vs_lowrank": lr_us / us, "speedup_vs_dense": dense_us / us, "weight_copies": copies}
    if decode:
        gbs = decode_bytes(T, m, n, r) / us / 1e3
        out["roofline"] = {"bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak,
                           "algorithmic_bytes_per_call": decode_bytes(T, m, n, r),
                           "peak_source": f"{peak_src} hbm_gbs"}
        out["lowrank_hbm_gbs"] = lowrank_bytes(T, m, n, r) / lr_us / 1e3
        out["dense_hbm_gbs"] = dense_bytes(T, m, n) / dense_us / 1e3
    else:
        tf = pifa_flops(T, m, n, r) / us / 1e6
        out["roofline"] = {"bound": "tensor", "achieved": tf, "peak": tc_peak, "unit": "TFLOP/s", "frac": tf / tc_peak,
                           "algorithmic_flops_per_call": pifa_flops(T, m, n, r),
                           "peak_source": f"{peak_src} bf16_tflops (burst)"}
        out["lowrank_tflops"] = 2 * T * r * (m + n) / lr_us / 1e6
        out["dense_tflops"] = 2 * T * m * n / dense_us / 1e6
    out["clocks"] = clk.summary()
    return out


# The library's selector (pifa_select_variant) runs the decode variant for T <= 64, and up to
# DECODE_MAX_T tokens where the non-pivot rows make 148 to 296 blocks of 128 and the pivot rows at
# most 296; the split prefill otherwise. is_decode restates it for the bench's workload names.
DECODE_MAX_T = 128


def is_decode(T, m, r, groups=1):
    if T <= 64:
        return True
    blocks_p, blocks_np = -(-groups * r // 128), -(-groups * (m - r) // 128)
    return T <= DECODE_MAX_T and blocks_p <= 296 and 148 <= blocks_np <= 296
DECODE_POINTS = [(inputs.ATTN7B, (1, 8, 16, 64)), (inputs.MLP7B_GATE, (1, 8, 16, 64)),
                 (inputs.MLP7B_DOWN, (1, 8, 16, 64)), (inputs.ATTN70B, (1, 8, 16, 64)),
                 (inputs.MLP70B_GATE, (1, 8, 16, 32, 64, 128))]
PREFILL_POINTS = [(inputs.ATTN7B, 2048), (inputs.ATTN7B, 8192), (inputs.ATTN70B, 4096), (inputs.MLP70B_GATE, 4096)]


def mlp7b_point(dev, stream, T, hbm_peak, tc_peak, peak_src):
    """The 7B MLP as three layers back to back per token batch (gate(X), up(X) on X of width 4096,
    down on an independent input of width 11008; no activation between them): three pifa_forward
    calls, and gate + up as one pifa_forward_grouped call followed by down, beside three low-rank
    and three dense layers; two weight copies of every layer (decode: enough to exceed L2)."""
    import torch
    from paper_2501_19090_gb300 import pifa as P
    G_, D_ = inputs.MLP7B_GATE, inputs.MLP7B_DOWN
    decode = is_decode(T, G_.m, G_.r)
    copies = 4 if decode else 2
    lay = {name: timing_layer(s, dev, seed, copies=copies) for name, s, seed in
           (("gate", G_, 1), ("up", G_, 2), ("down", D_, 3))}
    gen = torch.Generator(device=dev)
    gen.manual_seed(19)
    Xg = torch.randn((T, G_.n), device=dev, generator=gen).to(torch.bfloat16)
    Xd = torch.randn((T, D_.n), device=dev, generator=gen).to(torch.bfloat16)
    Y = {k: torch.empty((T, (G_ if k != "down" else D_).m), dtype=torch.bfloat16, device=dev) for k in lay}
    ws = P.workspace(max(P.pifa_workspace_size(T, s.m, s.n, s.r) for s in (G_, D_)), dev, tag="mlp")
    m, r = G_.m, G_.r
    piv_s = torch.cat([lay["gate"][0], lay["up"][0] + m])
    nonp_s = torch.cat([lay["gate"][1], lay["up"][1] + m])
    Wp_s = [torch.cat([lay["gate"][2][j], lay["up"][2][j]]) for j in range(copies)]
    C_s = [torch.cat([lay["gate"][3][j], lay["up"][3][j]]) for j in range(copies)]
    Yg = torch.empty((T, 2 * m), dtype=torch.bfloat16, device=dev)
    wsg = P.workspace(P.pifa_workspace_size_grouped(2, T, m, G_.n, r), dev, tag="mlpg")

    def three(i):
        j = i % copies
        for k, X in (("gate", Xg), ("up", Xg), ("down", Xd)):
            piv, nonp, Wps, Cs = lay[k]
            P.pifa_forward(X, Wps[j], Cs[j], piv, nonp, Y=Y[k], workspace_tensor=ws, stream=stream)

    def grouped(i):
        j = i % copies
        P.pifa_forward_grouped(2, Xg, Wp_s[j], C_s[j], piv_s, nonp_s, Y=Yg, workspace_tensor=wsg, stream=stream)
        piv, nonp, Wps, Cs = lay["down"]
        P.pifa_forward(Xd, Wps[j], Cs[j], piv, nonp, Y=Y["down"], workspace_tensor=ws, stream=stream)

    per = 16 if decode else 4
    with ClockSampler(torch.cuda.current_device()) as clk:
        us = _steady_us(three, per, stream)
        gus = _steady_us(grouped, per, stream)
        assert P.pifa_device_status(stream) == P.PIFA_OK
        del lay, Wp_s, C_s
        torch.cuda.empty_cache()
        cmp_ = {}
        for kind in ("lowrank", "dense"):
            fns = []
            for s in (G_, G_, D_):
                lr, dense, X = _comparator_fns(dev, s, T, gen, copies, 2)
                fns.append(lr if kind == "lowrank" else dense)
            cmp_[kind] = _steady_us(lambda i: [f(i) for f in fns], per, stream)
            del fns
            torch.cuda.empty_cache()
    shapes = (G_, G_, D_)
    out = {"workload": f"llama2_7b_mlp gate+up+down T={T}", "T": T, "us_per_step": us,
           "tokens_per_s": T / (us / 1e6), "grouped_us_per_step": gus, "grouped_tokens_per_s": T / (gus / 1e6),
           "lowrank_us": cmp_["lowrank"], "dense_us": cmp_["dense"],
           "speedup_vs_lowrank": cmp_["lowrank"] / min(us, gus), "speedup_vs_dense": cmp_["dense"] / min(us, gus)}
    if decode:
        b = sum(decode_bytes(T, s.m, s.n, s.r) for s in shapes)
        gbs = b / min(us, gus) / 1e3
        out["roofline"] = {"bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak,
                           "algorithmic_bytes_per_step": b, "peak_source": f"{peak_src} hbm_gbs"}
    else:
        f = sum(pifa_flops(T, s.m, s.n, s.r) for s in shapes)
        tf = f / min(us, gus) / 1e6
        out["roofline"] = {"bound": "tensor", "achieved": tf, "peak": tc_peak, "unit": "TFLOP/s", "frac": tf / tc_peak,
                           "algorithmic_flops_per_step": f, "peak_source": f"{peak_src} bf16_tflops (burst)"}
    out["clocks"] = clk.summary()
    return out


def backward_point(dev, stream, shape, T, tc_peak, peak_src):
    """pifa_backward (dX, dW_p, dC) at T tokens beside the same shape's dense backward (dX = dY W,
    dW = dY^T X) and two-factor low-rank backward (H = X V: dU = dY^T H, dH = dY U, dV = X^T dH,
    dX = dH V^T) through torch.matmul; tensor roofline on the PIFA backward's algorithmic FLOPs,
    2 T r (2 (m - r) + 2 n) (the Y_p recompute and the lo passes are not counted)."""
    import torch
    from paper_2501_19090_gb300 import pifa as P
    m, n, r = shape.m, shape.n, shape.r
    piv, nonp, Wps, Cs = timing_layer(shape, dev, 9, "bf16", 2)
    gen = torch.Generator(device=dev)
    gen.manual_seed(23)
    X = torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16)
    dY = torch.randn((T, m), device=dev, generator=gen).to(torch.bfloat16)
    ws = P.workspace(P.pifa_backward_workspace_size(T, m, n, r), dev, tag="bwd")
    torch.cuda.synchronize()

    def bwd(i):
        P.pifa_backward(X, Wps[i % 2], Cs[i % 2], piv, nonp, dY, workspace_tensor=ws, stream=stream)

    U = (torch.randn((m, r), device=dev, generator=gen) / math.sqrt(r)).to(torch.bfloat16)
    V = (torch.randn((n, r), device=dev, generator=gen) / math.sqrt(r)).to(torch.bfloat16)
    W = torch.randn((m, n), device=dev, generator=gen).to(torch.bfloat16)

    def dense(i):
        dY @ W
        dY.t() @ X

    def lowrank(i):
        H = X @ V
        dY.t() @ H
        dH = dY @ U
        X.t() @ dH
        dH @ V.t()

    with ClockSampler(torch.cuda.current_device()) as clk:
        us = _steady_us(bwd, 4, stream)
        assert P.pifa_device_status(stream) == P.PIFA_OK
        d_us = _steady_us(dense, 4, stream)
        l_us = _steady_us(lowrank, 4, stream)
    flops = 2 * T * r * (2 * (m - r) + 2 * n)
    tf = flops / us / 1e6
    del Wps, Cs, X, dY, U, V, W
    torch.cuda.empty_cache()
    return {"workload": f"{shape.name} backward T={T}", "us_per_call": us, "tokens_per_s": T / (us / 1e6),
            "dense_us": d_us, "lowrank_us": l_us, "speedup_vs_dense": d_us / us, "speedup_vs_lowrank": l_us / us,
            "roofline": {"bound": "tensor", "achieved": tf, "peak": tc_peak, "unit": "TFLOP/s", "frac": tf / tc_peak,
                         "algorithmic_flops_per_call": flops, "peak_source": f"{peak_src} bf16_tflops (burst)"},
            "clocks": clk.summary()}


def m_accumulate_point(dev, stream, shape, T, tc_peak, peak_src):
    """pifa_m_accumulate (X X^T and Y_t X^T of one calibration batch, lambda = 0.25) beside the same
    products through torch.matmul (bf16 in, fp32 out, X X^T whole); tensor roofline on
    T n (n + 1) + 4 T m n (the symmetric X X^T's upper triangle, Y_t = W X_mix^T, Y_t X^T)."""
    import torch
    from paper_2501_19090_gb300 import pifa as P
    m, n = shape.m, shape.n
    gen = torch.Generator(device=dev)
    gen.manual_seed(29)
    Xu = torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16)
    Xo = (Xu.float() + 0.1 * torch.randn((T, n), device=dev, generator=gen)).to(torch.bfloat16)
    W = (torch.randn((m, n), device=dev, generator=gen) / math.sqrt(n)).to(torch.bfloat16)
    XXt = torch.zeros((n, n), dtype=torch.float32, device=dev)
    YtXt = torch.zeros((m, n), dtype=torch.float32, device=dev)
    ws = P.workspace(P.pifa_m_accumulate_workspace_size(T, m, n), dev, tag="macc")
    torch.cuda.synchronize()

    def macc(i):
        P.pifa_m_accumulate(Xo, Xu, W, 0.25, XXt, YtXt, workspace_tensor=ws, stream=stream)

    def ref(i):
        XXt.add_((Xu.t() @ Xu).float())
        Yt = (0.25 * Xo.float() + 0.75 * Xu.float()).to(torch.bfloat16) @ W.t()
        YtXt.add_((Yt.t() @ Xu).float())

    with ClockSampler(torch.cuda.current_device()) as clk:
        us = _steady_us(macc, 4, stream)
        assert P.pifa_device_status(stream) == P.PIFA_OK
        t_us = _steady_us(ref, 4, stream)
    flops = T * n * (n + 1) + 4 * T * m * n
    tf = flops / us / 1e6
    del Xu, Xo, W, XXt, YtXt
    torch.cuda.empty_cache()
    return {"workload": f"{shape.name} M accumulators T={T}", "us_per_call": us, "tokens_per_s": T / (us / 1e6),
            "torch_us": t_us, "speedup_vs_torch": t_us / us,
            "torch_note": "single bf16 roundings of the mixed input and Y_t (the library carries them as hi + lo pairs)",
            "roofline": {"bound": "tensor", "achieved": tf, "peak": tc_peak, "unit": "TFLOP/s", "frac": tf / tc_peak,
                         "algorithmic_flops_per_call": flops, "peak_source": f"{peak_src} bf16_tflops (burst)"},
            "clocks": clk.summary()}


def extras(dev, stream, hbm_peak, tc_peak, peak_src):
    """Every configuration of the workload list beside its low-rank and dense layers (one GPU)."""
    import torch
    out = {"decode_points": [], "mlp7b_three_layers": [], "prefill_points": [], "rank_sweep": []}
    for shape, Ts in DECODE_POINTS:
        for T in Ts:
            out["decode_points"].append(layer_point(dev, stream, shape, T, hbm_peak, tc_peak, peak_src))
    for T in (1, 2048):
        out["mlp7b_three_layers"].append(mlp7b_point(dev, stream, T, hbm_peak, tc_peak, peak_src))
    for shape, T in PREFILL_POINTS:
        out["prefill_points"].append(layer_point(dev, stream, shape, T, hbm_peak, tc_peak, peak_src))
    for s in inputs.rank_sweep_shapes():
        out["rank_sweep"].append(layer_point(dev, stream, s, 2048, hbm_peak, tc_peak, peak_src))
    out["backward"] = [backward_point(dev, stream, sh, 2048, tc_peak, peak_src)
                       for sh in (inputs.ATTN7B, inputs.MLP7B_GATE)]
    out["m_accumulate"] = [m_accumulate_point(dev, stream, inputs.ATTN7B, 2048, tc_peak, peak_src)]
    torch.cuda.empty_cache()
    return out


def _pifa_c_dtype(c_dtype):
    from paper_2501_19090_gb300 import pifa as P
    return P.PIFA_DTYPE_FP16 if c_dtype == "fp16" else P.PIFA_DTYPE_BF16


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
    K = max(1, args.steps)
    decode = is_decode(T, m, r)
    wbytes = 2 * r * (m + n - r)
    copies = _copies_for(dev, wbytes)
    piv, nonp, Wps, Cs = timing_layer(shape, dev, 0, args.c_dtype, copies)
    gen = torch.Generator(device=dev)
    gen.manual_seed(1 + rank)
    Xs = [torch.randn((T, n), device=dev, generator=gen).to(torch.bfloat16) for _ in range(copies)]
    Ys = [torch.empty((T, m), dtype=torch.bfloat16, device=dev) for _ in range(copies)]
    cdt = _pifa_c_dtype(args.c_dtype)
    variant = P.pifa_select_variant(T, m, n, r, cdt)
    ws = P.workspace(P.pifa_workspace_size(T, m, n, r, variant, cdt), dev)
    stream = torch.cuda.Stream(device=dev)

    def step(i):
        j = i % copies
        P.pifa_forward(Xs[j], Wps[j], Cs[j], piv, nonp, Y=Ys[j], variant=variant, workspace_tensor=ws,
                       stream=stream)

    # W untimed warm-up steps (eager), then graphs covering exactly K steps: `reps` replays of a
    # graph of `per` steps plus one graph of the remainder
    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            step(i)
    stream.synchronize()
    assert P.pifa_device_status(stream) == P.PIFA_OK
    # kernels one step enqueues, counted by the library itself
    c0 = P.pifa_launch_count()
    with torch.cuda.stream(stream):
        step(0)
    launches_per_step = P.pifa_launch_count() - c0
    stream.synchronize()
    per = min(K, copies * max(1, 64 // copies))
    g = _graph_of(step, per, stream)
    reps, rem = divmod(K, per)
    g_rem = _graph_of(step, rem, stream) if rem else None

    def region():
        for _ in range(reps):
            g.replay()
        if g_rem is not None:
            g_rem.replay()

    with torch.cuda.stream(stream):          # replays launch on the current stream
        for _ in range(max(3, args.warmup)):
            region()
    stream.synchronize()

    dist = _dist()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)

    def timed_region():
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            e0.record(stream)
            region()
            e1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        return _max_over_ranks(e0.elapsed_time(e1))

    # The timed region (exactly K steps) is repeated until ~0.3 s have passed, so that the clock
    # sampler sees it; value comes from the median repetition.
    first = timed_region()
    n_rep = max(3, min(2000, math.ceil(0.3 / max(first / 1e3, 1e-6))))
    with ClockSampler(local_rank) as clk:
        times = [timed_region() for _ in range(n_rep)]
    st = P.pifa_device_status(stream)
    assert st == P.PIFA_OK, P.pifa_status_string(st)
    ms_region = statistics.median(times)
    step_ms = ms_region / K
    value = _job_value(world, T, K, ms_region)
    del g, g_rem

    # --- e2e through the public API with pinned host buffers ---
    nh = 4
    Xhs = [torch.empty((T, n), dtype=torch.bfloat16).pin_memory() for _ in range(nh)]
    for i in range(nh):
        Xhs[i].copy_(Xs[i % copies].cpu())
    e2e_steps = max(64, min(4000, math.ceil(0.3 / max(step_ms / 1e3, 1e-7))))
    e2e_pipe, e2e_pipe_steps, e2e_pipe_per = e2e_pipelined(P, dev, T, n, m, Xhs, Wps, Cs, piv, nonp, variant, ws,
                                                           stream, world, e2e_steps)
    e2e_serial = e2e_serial_graph(P, dev, T, n, m, Xhs, Wps, Cs, piv, nonp, variant, ws, stream, world, e2e_steps)

    ab = decode_bytes(T, m, n, r)
    af = pifa_flops(T, m, n, r)
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{shape.name} {'decode' if decode else 'prefill'} T={T}", "m": m, "n": n, "r": r,
                   "tokens_per_step": T, "c_dtype": args.c_dtype, "variant": P.pifa_variant_name(variant),
                   "parallelism": f"replicas{world}",
                   "operands": "seeded synthetic layer: random ascending pivot set, W_p ~ N(0, 1/r), C ~ N(0, 0.18^2), "
                               "X ~ N(0, 1), all bf16 (kernel time does not depend on the values)",
                   "l2_defeat": f"{copies} rotating weight copies with their own X and Y "
                                f"({copies * wbytes / 1e6:.0f} MB > 3x L2)",
                   "timing": f"exactly {K} steps per timed region (CUDA graph replays, CUDA events on the launching "
                             f"stream); the region repeated {n_rep} times, value from the median"},
        "timed_repeats": n_rep,
        "e2e": {"value": e2e_pipe, "unit": "tokens/s", "h2d_bytes_per_step": T * n * 2,
                "d2h_bytes_per_step": T * m * 2,
                "mode": f"serving loop: per step X uploaded from pinned host memory (one copy per step), "
                        f"pifa_forward, Y downloaded to pinned host memory (one copy per step); steps in groups of "
                        f"4 with two groups in flight, uploads and downloads on two copy streams overlapping the "
                        f"neighbouring groups' forwards, the compute stream waiting on the copies once per group; "
                        f"{e2e_pipe_per} steps per CUDA graph, {e2e_pipe_steps} steps timed; the last step's Y "
                        f"checked against a separate forward",
                "serial_value": e2e_serial,
                "serial_mode": "the same steps one after another on one stream (upload, forward, download), "
                               "captured as a CUDA graph and replayed"},
        "roofline": ({"bound": "hbm", "achieved": ab / (step_ms / 1e3) / 1e9, "peak": hbm_peak, "unit": "GB/s",
                      "frac": ab / (step_ms / 1e3) / 1e9 / hbm_peak,
                      "traffic": _traffic(shape.name, T),
                      "peak_source": f"{peak_src} hbm_gbs (burst: the call is timed alone)",
                      "kernel": f"decode phase 1 + phase 2 ({launches_per_step} PDL-chained kernels per call)",
                      "algorithmic_bytes_per_launch": ab} if decode else
                     {"bound": "tensor", "achieved": af / (step_ms / 1e3) / 1e12, "peak": tc_peak,
                      "unit": "TFLOP/s", "frac": af / (step_ms / 1e3) / 1e12 / tc_peak,
                      "traffic": None, "peak_source": f"{peak_src} bf16_tflops (burst)",
                      "kernel": f"{P.pifa_variant_name(variant)} prefill (GEMM 1 + GEMM 2 per call)",
                      "algorithmic_flops_per_launch": af}),
        "gpu_launches": K * launches_per_step,
        "gpu_launches_per_step": launches_per_step,
        "gpu_launches_all_repeats": K * launches_per_step * n_rep,
        "clocks": clk.summary(),
    }
    del Wps, Cs, Xs, Ys
    torch.cuda.empty_cache()
    if rank == 0 and world == 1 and not args.no_extras and shape is SHAPE and T == T_DECODE:
        # one GPU only (at N > 1 every GPU would wait for rank 0's extras)
        out["comparators"] = layer_point(dev, stream, shape, T, hbm_peak, tc_peak, peak_src,
                                         name="headline layer, same T (PIFA re-timed beside the comparators)")
        out.update(extras(dev, stream, hbm_peak, tc_peak, peak_src))
        out["cpu_baseline"] = cpu_baseline(shape, T)
    return out


def e2e_serial_graph(P, dev, T, n, m, Xhs, Wps, Cs, piv, nonp, variant, ws, stream, world, steps):
    """The serial serving loop (upload X, forward, download Y, one after another on one stream)
    captured as a CUDA graph and replayed; tokens/s over all ranks."""
    import torch
    nh = len(Xhs)
    copies = len(Wps)
    Xd = torch.empty((T, n), dtype=torch.bfloat16, device=dev)
    Yd = torch.empty((T, m), dtype=torch.bfloat16, device=dev)
    Yhs = [torch.empty((T, m), dtype=torch.bfloat16).pin_memory() for _ in range(nh)]

    def e2e_step(i):
        Xd.copy_(Xhs[i % nh], non_blocking=True)
        P.pifa_forward(Xd, Wps[i % copies], Cs[i % copies], piv, nonp, Y=Yd, variant=variant, workspace_tensor=ws,
                       stream=stream)
        Yhs[i % nh].copy_(Yd, non_blocking=True)

    per = copies * max(1, 64 // copies)
    g = _graph_of(e2e_step, per, stream)
    reps = max(1, steps // per)
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
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    return _job_value(world, T, reps * per, _max_over_ranks(e0.elapsed_time(e1)))


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


def _host_layer(shape, seed=0):
    """The headline layer's operands on the host for the oracle timings: inputs.synthetic_layer of
    the shape (random ascending pivots, W_p ~ N(0, 1/r), C ~ N(0, 0.18^2), bf16 values). The
    oracle's time depends on the shapes only."""
    piv, nonp, Wp, C = inputs.synthetic_layer(shape.m, shape.n, shape.r, seed)
    return piv.astype(np.int64), nonp.astype(np.int64), Wp.astype(np.float64), C.astype(np.float64)


def cpu_baseline(shape, T, budget_s=10.0, single_s=5.0):
    """The fp64 oracle forward (numpy) on the host cores over a bounded sample of the workload,
    with BLAS_THREADS BLAS threads; the same forward on one thread, timed in a fresh interpreter
    (numpy's thread count is fixed when it loads), is reported beside it."""
    import oracle
    piv, nonp, Wp, C = _host_layer(shape)
    rng = np.random.default_rng(9)
    X = inputs.make_activations(rng, T, shape.n, "bf16")
    oracle.forward(X, Wp, C, piv, nonp)
    t0 = time.perf_counter()
    calls = 0
    while time.perf_counter() - t0 < budget_s:
        oracle.forward(X, Wp, C, piv, nonp)
        calls += 1
    dt = time.perf_counter() - t0
    out = {"value": calls * T / dt, "unit": "tokens/s", "cores": BLAS_THREADS, "kind": "oracle",
           "sample": f"{calls} oracle forwards of T={T} tokens on {shape.name} (fp64 numpy, "
                     f"{BLAS_THREADS} BLAS threads), {dt:.1f} s"}
    try:
        out["single_thread"] = _oracle_rate_one_thread(shape, T, single_s)
    except Exception as e:  # reported, never fatal: the main figure stands on its own
        out["single_thread"] = {"error": f"{type(e).__name__}: {e}"}
    return out


_ONE_THREAD_TIMER = """
import json, sys, time
import numpy as np
sys.path.insert(0, sys.argv[1])
import oracle
from paper_2501_19090_gb300 import inputs
m, n, r, T = (int(v) for v in sys.argv[2:6])
piv, nonp, Wp, C = inputs.synthetic_layer(m, n, r, 0)
args = (inputs.make_activations(np.random.default_rng(9), T, n, "bf16"), Wp.astype(np.float64),
        C.astype(np.float64), piv.astype(np.int64), nonp.astype(np.int64))
oracle.forward(*args)
t0, calls = time.perf_counter(), 0
while time.perf_counter() - t0 < float(sys.argv[6]):
    oracle.forward(*args)
    calls += 1
print(json.dumps({"calls": calls, "seconds": time.perf_counter() - t0}))
"""


def _oracle_rate_one_thread(shape, T, budget_s):
    """Tokens/s of the oracle forward with one BLAS thread, in a fresh interpreter."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-c", _ONE_THREAD_TIMER, ROOT, str(shape.m), str(shape.n), str(shape.r),
                        str(T), str(budget_s)], env=env, capture_output=True, text=True, timeout=budget_s + 180)
    if r.returncode != 0:
        raise RuntimeError(r.stderr.strip().splitlines()[-1] if r.stderr.strip() else f"exit {r.returncode}")
    res = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": res["calls"] * T / res["seconds"], "unit": "tokens/s", "cores": 1,
            "sample": f"{res['calls']} oracle forwards, {res['seconds']:.1f} s, one BLAS thread"}


def _traffic(layer, T):
    t = NCU_TRAFFIC.get((layer, T))
    if not t or any(_src_sha(f) != h for f, h in t["sha"].items()):
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
    """Reference arm: the fp64 oracle (the paper publishes no code) on the host cores, on the same
    workload as our arm's line (rank 0 only; other ranks exit without work)."""
    import oracle
    if rank != 0:
        return None
    shape = SHAPES[args.shape]
    T = args.tokens
    piv, nonp, Wp, C = _host_layer(shape)
    rng = np.random.default_rng(1)
    X = inputs.make_activations(rng, T, shape.n, "bf16")
    for _ in range(max(3, args.warmup)):
        oracle.forward(X, Wp, C, piv, nonp)
    # bounded sample: at most ~60 s of oracle forwards, however many steps were asked for
    t0 = time.perf_counter()
    done = 0
    while done < args.steps and (done == 0 or time.perf_counter() - t0 < 60.0):
        oracle.forward(X, Wp, C, piv, nonp)
        done += 1
    dt = time.perf_counter() - t0
    v = T * done / dt
    cores = BLAS_THREADS
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": done, "requested_steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / done,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": f"{shape.name} {'decode' if is_decode(T, shape.m, shape.r) else 'prefill'} T={T}",
                                            "m": shape.m, "n": shape.n, "r": shape.r, "tokens_per_step": T,
                                            "c_dtype": args.c_dtype, "parallelism": f"replicas{args.gpus}"},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{done} of {args.steps} requested fp64 oracle forwards of T={T} on a seeded "
                                       f"synthetic layer of the shape (numpy, {cores} BLAS threads; capped at ~60 s)"},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    global _DIST
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--tokens", type=int, default=T_DECODE)
    ap.add_argument("--no-extras", action="store_true")
    ap.add_argument("--c-dtype", default="bf16", choices=["bf16", "fp16"])
    ap.add_argument("--shape", default=SHAPE.name, choices=sorted(SHAPES),
                    help="layer shape of the main line (extras run with the default shape and T only)")
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
