"""Benchmark of the RoLA attention layer on GB300.

One step = one pass of the whole module (block mask, low-rank summary, sparse
branch, readout + fusion) over one Wan2.1-14B 720p-shaped layer (B=1, 40 heads,
21 x 45 x 80 = 75600 tokens, d_h=128, 90 % block sparsity, r=32) with seeded
synthetic bf16 inputs already resident in HBM.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload wan14b_720p] [--no-dense] [--no-cpu]

Under torchrun each rank runs its own replica layer (the module shards by
(batch, head) with no exchange, so there is no data-path collective); value is
the tokens of all ranks divided by the slowest rank's time.
`--impl reference` times the fp64 CPU oracle on a bounded sample of the same
workload on the host cores (rank 0 only).
"""
from __future__ import annotations

import argparse
import csv
import io
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

METRIC = "RoLA attn layer ms & tokens/s (Wan2.1-14B 720p shape); % of TC/HBM roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# The ncu summary that carries the sparse kernel's DRAM traffic per (head, token), and
# the sources its capture was taken on.
SPARSE_PROFILE = os.path.join(ROOT, "profiles", "sparse_attn_rows_wan13b_480p.md")
SPARSE_SOURCES = ["sparse_attn_rows.cu", "common.cuh", "tcgen05.cuh", "tensor_map.cuh"]


def sparse_traffic_per_head_token():
    """dram__bytes_read.sum + dram__bytes_write.sum of the sparse kernel per (head, token),
    from the committed ncu summary, or None when the kernel's sources have changed since
    that capture (their sha256 no longer matches the one the summary records)."""
    import hashlib
    try:
        text = open(SPARSE_PROFILE).read()
    except OSError:
        return None
    fields = dict(line.split(": ", 1) for line in text.splitlines()
                  if line.startswith(("traffic_bytes_per_head_token: ", "kernel_sources_sha256: ")))
    if len(fields) != 2:
        return None
    h = hashlib.sha256()
    for f in SPARSE_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_06712_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    if h.hexdigest() != fields["kernel_sources_sha256"].strip():
        return None
    return float(fields["traffic_bytes_per_head_token"])


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------- accounting

def block_sizes(cfg, block=64):
    """Tokens per block: 64-token chunks (the last one ragged), or the real tokens of each
    4 x 4 x 4 cube of the latent grid (edge cubes hold fewer)."""
    if cfg.get("block_geometry", "flat") == "cube":
        ext = lambda n: [min(4, n - 4 * c) for c in range(-(-n // 4))]
        return [a * b * c for a in ext(cfg["T"]) for b in ext(cfg["Hh"]) for c in ext(cfg["Ww"])]
    nB = -(-cfg["N"] // block)
    return [block] * (nB - 1) + [cfg["N"] - (nB - 1) * block]


def sparse_flops_from_mask(kv_idx, sizes, d_h=128, qsizes=None):
    """Algorithmic FLOPs of the sparse branch: 4 d_h sum_{h,i} |Q_i| sum_{j kept} |K_j|
    (QK^T and PV, 2 flops per multiply-add), every block counted at its real size
    (App. D, C_sparse = 4 B H L^2 (1-S) d_h).  qsizes: the query blocks' sizes when they
    differ from the key blocks' (128-token query chunks)."""
    import torch
    sizes = torch.tensor(sizes, dtype=torch.float64, device=kv_idx.device)
    qs = sizes if qsizes is None else torch.tensor(qsizes, dtype=torch.float64, device=kv_idx.device)
    keys = sizes[kv_idx.long()].sum(dim=-1)            # [B,H,nQB] kept keys per query block
    return float(4.0 * d_h * (keys * qs).sum().item())


def lowrank_flops(B, H, N, d_h, r):
    """App. D: C_lowrank = 8 B H L d_h r (projections, context, readout)."""
    return 8.0 * B * H * N * d_h * r


# kernels one bf16 forward launches: RoPE table, fused pre-pass, block scores,
# top-k, summary combine, sparse attention, readout + fusion; with cube blocks
# the pre-pass splits into the cube rotate + pool and the summary-only pre-pass
LAUNCHES_PER_FORWARD = {"flat": 7, "cube": 8}


def summary_bytes(B, H, N, d_h, esize=2):
    """HBM bytes the summary must move: read k and v once."""
    return 2.0 * B * H * N * d_h * esize


# ----------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.tmp = None

    def start(self):
        try:
            self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.tmp, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.tmp.flush()
        self.tmp.seek(0)
        rows = [r for r in csv.reader(io.StringIO(self.tmp.read())) if len(r) >= 9]
        os.unlink(self.tmp.name)
        sm, smax, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                smax.append(float(r[2]))
                power.append(float(r[3]))
            except ValueError:
                continue
            for nm, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        load = [x for x in sm if x > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(load), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power) if power else None}


# ----------------------------------------------------------------- CPU oracle baseline

def oracle_sample_time(cfg, heads, qblocks):
    """Wall time of the oracle forward on `heads` heads of the layer and the given
    query blocks (mask, summary and RoPE over the whole sequence of those heads)."""
    import torch
    from oracle import oracle as O
    from paper_2609_06712_gb300 import inputs
    sub = dict(cfg, H=heads)
    x = inputs.make_inputs(sub, dtype=torch.bfloat16)
    h = {k: (None if v is None else v.float().numpy()) for k, v in x.items()}
    t0 = time.perf_counter()
    O.forward(sub, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], qblocks=qblocks)
    return time.perf_counter() - t0


def cpu_oracle_estimate(cfg, heads=None, q_lo=8, q_hi=96):
    """Layer time of the oracle extrapolated from a bounded sample: `heads` heads in
    parallel with q_lo and q_hi query blocks each; the difference gives the
    per-query-block cost, the rest the per-head fixed cost (mask, summary)."""
    from oracle import oracle as O
    O.build()
    cores = os.cpu_count() or 1
    heads = heads or min(cfg["H"], cores)
    nB = len(block_sizes(cfg, cfg["block"]))
    t_lo = oracle_sample_time(cfg, heads, list(range(q_lo)))
    t_hi = oracle_sample_time(cfg, heads, list(range(q_hi)))
    per_block = max(t_hi - t_lo, 0.0) / (q_hi - q_lo)
    fixed = max(t_lo - q_lo * per_block, 0.0)
    layer_s = (cfg["H"] / heads) * (fixed + nB * per_block)
    tokens_s = cfg["B"] * cfg["N"] / layer_s
    sample = (f"fp64 oracle on {heads} of {cfg['H']} heads (full-sequence mask, RoPE and summary) with "
              f"{q_lo} and {q_hi} of {nB} query blocks; layer time extrapolated per query block and per head")
    return {"value": tokens_s, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample,
            "layer_s_est": layer_s, "sample_s": t_lo + t_hi}


# ----------------------------------------------------------------- main

def dist_setup(args):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return ws, rank, local


def reduce_max(x, ws):
    """Largest value over the ranks (the slowest rank's time); x itself for one rank."""
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank, ms_per_step_max, ws):
    """Whole-job tokens/s: every rank runs its own layer replica (weak scaling), so the
    job processes ws * tokens_per_rank tokens per step in the slowest rank's time."""
    return ws * tokens_per_rank / (ms_per_step_max * 1e-3)


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def run_reference(args, cfg, ws, rank):
    if rank != 0:
        return
    from oracle import oracle as O
    O.build()
    times = []
    est = None
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        est = cpu_oracle_estimate(cfg, q_lo=1, q_hi=3)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    line = {
        "impl": "reference", "metric": METRIC, "value": est["value"], "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * est["layer_s_est"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": cfg["name"], "B": cfg["B"], "H": cfg["H"], "N": cfg["N"],
                   "grid": [cfg["T"], cfg["Hh"], cfg["Ww"]], "keep": cfg["keep"], "r": cfg["r"],
                   "lowrank_act": cfg.get("lowrank_act", "silu")},
        "cpu_baseline": {"value": est["value"], "unit": "tokens/s", "cores": est["cores"], "kind": "oracle",
                         "sample": est["sample"], "wall_s_per_step": statistics.median(times)},
        "e2e": {"value": est["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# fp32 FMA peak of the SIMT backward kernels: 152 SMs x 128 fp32 lanes x 2 flops x 2.07 GHz
FP32_SIMT_PEAK_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def run_backward(args, cfg, c, x, stream, ws, rank):
    """Times rola_forward_train and rola_backward (one training step of the module) on the layer."""
    import torch
    from paper_2609_06712_gb300 import rola
    dev = x["q"].device
    B, H, N, r = cfg["B"], cfg["H"], cfg["N"], cfg["r"]
    wsb = rola.workspace(c, dev)
    bws = rola.backward_workspace(c, dev)
    o, o_s = torch.empty_like(x["q"]), torch.empty_like(x["q"])
    kv = torch.empty((B, H, rola.num_blocks(c), rola.num_keep(c)), dtype=torch.int32, device=dev)
    lse = torch.empty((B, H, N), dtype=torch.float32, device=dev)
    C = torch.empty((B, H, r, 128), dtype=torch.float32, device=dev)
    dO = torch.randn(x["q"].shape, generator=torch.Generator(device=dev).manual_seed(5), device=dev,
                     dtype=torch.float32).to(x["q"].dtype)
    g = {n: torch.empty_like(x[n[1:]]) for n in ("dq", "dk", "dv")}
    dPq = torch.empty(x["P_q"].shape, dtype=torch.float32, device=dev)
    dPk = torch.empty(x["P_k"].shape, dtype=torch.float32, device=dev)
    dgate = torch.empty((B, N), dtype=torch.float32, device=dev) if x["gate"] is not None else None
    fw = lambda: rola.forward_train(c, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], o, kv, o_s, lse, C,
                                    wsb)
    bw = lambda: rola.backward(c, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], kv, o_s, lse, C, dO,
                               g["dq"], g["dk"], g["dv"], dPq, dPk, dgate, bws)
    for _ in range(args.warmup):
        fw()
        bw()
    torch.cuda.synchronize()
    barrier(ws)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    t_fw = t_bw = 0.0
    for _ in range(args.steps):
        ev[0].record(stream)
        fw()
        ev[1].record(stream)
        bw()
        ev[2].record(stream)
        torch.cuda.synchronize()
        t_fw += ev[0].elapsed_time(ev[1])
        t_bw += ev[1].elapsed_time(ev[2])
    ms_fw = reduce_max(t_fw / args.steps, ws)
    ms_bw = reduce_max(t_bw / args.steps, ws)
    assert rola.get_device_status(wsb) == rola.ROLA_OK and rola.get_device_status(bws) == rola.ROLA_OK
    if rank == 0:
        sparse_fw = sparse_flops_from_mask(kv, block_sizes(cfg))
        # algorithmic: recompute S, dP = dO^s V^T, dQ, dK, dV (5 products of the sparse pattern), and the
        # low-rank backward's six N x r x d_h products (u, y, dq~, dq, dC, dP_q on the query side; u, dk~,
        # dv, dk, dP_k on the key side: 11 products of 2 N d_h r flops)
        flops = 2.5 * sparse_fw + 11 * 2.0 * B * H * N * 128 * r
        if c.dtype == rola.ROLA_BF16:
            # the sparse gradient products run on the tcgen05 tensor cores (fp32 accumulation in TMEM),
            # the low-rank ones on mma.sync
            peaks, src = load_peaks()
            peak = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
            bound, peak_src = "tensor", f"{src} bf16_tflops_sustained"
        else:
            peak, bound = FP32_SIMT_PEAK_TFLOPS, "alu"
            peak_src = "fp32 FMA lanes x clock (152 SMs x 128 x 2 x 2.07 GHz), derived"
        print(json.dumps({"entry": "rola_backward", "ms_forward_train": ms_fw, "ms_backward": ms_bw,
                          "train_step_tokens_per_s": job_throughput(B * N, ms_fw + ms_bw, ws),
                          "backward_flops": flops, "achieved_tflops": flops / (ms_bw * 1e-3) / 1e12,
                          "bound": bound, "peak_tflops": peak,
                          "frac": flops / (ms_bw * 1e-3) / 1e12 / peak, "peak_source": peak_src,
                          "steps": args.steps, "warmup": args.warmup,
                          "config": {"workload": cfg["name"], "B": B, "H": H, "N": N, "r": r, "keep": cfg["keep"],
                                     "dtype": "bf16"}}), flush=True)


def run_entry(args, cfg, c, x, o, kv, wsb, stream, ws, rank):
    """Times one per-stage entry point of the C ABI on the layer (inputs resident in HBM)."""
    import torch
    from paper_2609_06712_gb300 import rola
    C = torch.empty((cfg["B"], cfg["H"], cfg["r"], 128), dtype=torch.float32, device=o.device)
    rola.forward(c, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], o, kv, wsb)    # a mask and O^s to use
    tensor_bytes = 2.0 * cfg["B"] * cfg["H"] * cfg["N"] * 128
    calls = {
        "mask": (lambda: rola.block_mask(c, x["q"], x["k"], kv, wsb), 4 * tensor_bytes,
                 "read q, k; write q^r, k^r (rotate + pool), then scores and top-k"),
        "summary": (lambda: rola.lowrank_summary(c, x["k"], x["v"], x["P_k"], C, None, wsb), 2 * tensor_bytes,
                    "read k, v"),
        "sparse": (lambda: rola.sparse_attn(c, x["q"], x["k"], x["v"], kv, o, wsb), 6 * tensor_bytes,
                   "rotate q, k (read q, k; write q^r, k^r), then the sparse kernel (read q^r, k^r, v; write O^s)"),
        "apply": (lambda: rola.lowrank_apply(c, x["q"], x["P_q"], C, x["gate"], o, o, wsb), 3 * tensor_bytes,
                  "read q, O^s; write O"),
    }
    if args.entry == "out_proj":
        d_model = cfg["H"] * 128
        wo = (torch.randn((d_model, d_model), device=o.device) / d_model ** 0.5).to(torch.bfloat16)
        bo = 0.1 * torch.randn((d_model,), device=o.device)
        ybuf = torch.empty((cfg["B"], cfg["N"], d_model), dtype=torch.bfloat16, device=o.device)
        calls["out_proj"] = (lambda: rola.out_proj(c, o, wo, bo, ybuf, wsb),
                             tensor_bytes + 2.0 * d_model * d_model + 2.0 * cfg["B"] * cfg["N"] * d_model,
                             "Y = concat_h(O) W_o^T + b_o (tcgen05 GEMM): read O, W_o; write Y")
    fn, nbytes, what = calls[args.entry]
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    barrier(ws)
    a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(args.steps):
        fn()
    z.record(stream)
    torch.cuda.synchronize()
    ms = reduce_max(a.elapsed_time(z) / args.steps, ws)
    assert rola.get_device_status(wsb) == rola.ROLA_OK
    if rank == 0:
        peaks, src = load_peaks()
        hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
        names = {"mask": "rola_block_mask", "summary": "rola_lowrank_summary", "sparse": "rola_sparse_attn",
                 "apply": "rola_lowrank_apply", "out_proj": "rola_out_proj"}
        extra = {}
        if args.entry == "out_proj":
            fl = 2.0 * cfg["B"] * cfg["N"] * (cfg["H"] * 128) ** 2
            bf16_peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
            extra = {"flops_per_call": fl, "achieved_tflops": fl / (ms * 1e-3) / 1e12, "bf16_peak_tflops": bf16_peak,
                     "frac_of_burst": fl / (ms * 1e-3) / 1e12 / bf16_peak}
        print(json.dumps({"entry": names[args.entry], "ms_per_call": ms, "unit": "ms", "steps": args.steps, "warmup": args.warmup,
                          **extra,
                          "bytes_per_call": nbytes, "achieved_gbs": nbytes / (ms * 1e-3) / 1e9, "hbm_peak_gbs": hbm,
                          "note": what, "config": {"workload": cfg["name"], "H": cfg["H"], "N": cfg["N"],
                                                   "r": cfg["r"], "keep": cfg["keep"]}}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="wan14b_720p")
    ap.add_argument("--keep", type=float, default=None)
    ap.add_argument("--r", type=int, default=None)
    ap.add_argument("--geometry", default=None, choices=["flat", "cube"],
                    help="blocks of the sparse branch: 64-token chunks (default) or 4x4x4 cubes of the latent grid")
    ap.add_argument("--lowrank-act", default=None, choices=["silu", "identity", "tanh", "relu", "gelu"],
                    help="feature map of the low-rank branch (the activation ablation); default SiLU")
    ap.add_argument("--qblock", type=int, default=None, choices=[64, 128],
                    help="tokens per query block of the mask (128: the b_q = 128 variant); default 64")
    ap.add_argument("--no-dense", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--entry", default="forward", choices=["forward", "mask", "summary", "sparse", "apply", "out_proj",
                                                           "backward"],
                    help="time one per-stage entry point alone instead of the layer")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    from paper_2609_06712_gb300 import configs
    over = {}
    if args.keep is not None:
        over["keep"] = args.keep
    if args.r is not None:
        over["r"] = args.r
    if args.workload == "sweep":          # the rank x sparsity sweep at the 720p shape (seed of the sweep)
        cfg = configs.sweep_config(args.r if args.r is not None else 32, args.keep if args.keep is not None else 0.1)
    else:
        cfg = configs.get(args.workload, **over)
    if args.lowrank_act is not None:
        cfg["lowrank_act"] = args.lowrank_act
    if args.geometry is not None:
        cfg["block_geometry"] = args.geometry
    if args.qblock is not None:
        cfg["qblock"] = args.qblock
    ws, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, cfg, ws, rank)
        return

    import torch
    from paper_2609_06712_gb300 import build as rbuild
    rbuild.build()
    from paper_2609_06712_gb300 import inputs, rola

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    x = inputs.make_inputs(cfg, dtype=torch.bfloat16, device=dev, seed=cfg["seed"] + 1000 * rank)
    c = rola.make_config(cfg)
    wsb = rola.workspace(c, dev)
    nB, nk = rola.num_blocks(c), rola.num_keep(c)
    o = torch.empty_like(x["q"])
    kv = torch.empty((cfg["B"], cfg["H"], rola.num_query_blocks(c), nk), dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    K = args.steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(K)]
    for row in evs:
        for e in row:
            e.record(stream)
    args_fw = (c, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], o, kv, wsb)
    if args.entry == "backward":
        run_backward(args, cfg, c, x, stream, ws, rank)
        return
    if args.entry != "forward":
        run_entry(args, cfg, c, x, o, kv, wsb, stream, ws, rank)
        return

    for _ in range(args.warmup):
        rola.forward(*args_fw)
    torch.cuda.synchronize()
    assert rola.get_device_status(wsb) == rola.ROLA_OK

    # ---- device-timed region: inputs resident in HBM (each of q, k, v > L2)
    clocks = ClockSampler(local)
    barrier(ws)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for i in range(K):
        rola.forward_timed(*args_fw, evs[i])
    stop.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier(ws)
    ms_total = start.elapsed_time(stop)
    ms_step = reduce_max(ms_total / K, ws)
    # bf16 stages: one pass over q, k, v (rotation, block means, summary partials);
    # block scores + top-k + summary combine; sparse branch; readout + fusion
    stage_names = ["prepass", "select", "sparse_attn", "apply_fuse"]
    stage_ms = {n: statistics.mean(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(K))
                for j, n in enumerate(stage_names)}
    per_step = sorted(evs[i][0].elapsed_time(evs[i][4]) for i in range(K))
    step_stats = {"median": statistics.median(per_step), "min": per_step[0],
                  "p90": per_step[min(K - 1, int(round(0.9 * (K - 1))))]}
    assert rola.get_device_status(wsb) == rola.ROLA_OK
    tokens = cfg["B"] * cfg["N"]
    value = job_throughput(tokens, ms_step, ws)

    # ---- roofline of the dominant kernel (the sparse branch: tensor-core bound)
    peaks, peak_src = load_peaks()
    geometry = cfg.get("block_geometry", "flat")
    fl = sparse_flops_from_mask(kv, block_sizes(cfg),
                                qsizes=block_sizes(cfg, 128) if cfg.get("qblock", 0) == 128 else None)
    sp_ms = stage_ms["sparse_attn"]
    achieved = fl / (sp_ms * 1e-3) / 1e12
    # burst peak: the timed region is well under a second and ran at full SM clock (the
    # sustained figure was measured over 4 s under the power cap, at a lower clock)
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    peak_sus = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    # the capture is of the 64-token query blocks on contiguous key blocks
    tph = sparse_traffic_per_head_token() if geometry == "flat" and cfg.get("qblock", 0) in (0, 64) else None
    traffic = None if tph is None else tph * cfg["B"] * cfg["H"] * cfg["N"]
    roofline = {"bound": "tensor", "kernel": "sparse_attn", "achieved": achieved, "peak": peak,
                "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
                "peak_source": f"{peak_src} bf16_tflops (burst: sub-second timed region at full clock)",
                "frac_of_sustained": achieved / peak_sus,
                "traffic_source": (None if traffic is None else
                                   "profiles/sparse_attn_rows_wan13b_480p.md, per (head, token) x B*H*N"),
                "algorithmic_flops_per_launch": fl, "ms_per_launch": sp_ms}
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    tensor_bytes = summary_bytes(cfg["B"], cfg["H"], cfg["N"], 128) / 2      # one [B,H,N,128] bf16 tensor
    pre_bytes = 5 * tensor_bytes                                                # read q, k, v; write q^r, k^r
    pre_note = ("bytes = read q, k, v once + write the rotated q^r, k^r the sparse branch reads; "
                "algorithmic_bytes = the reads alone")
    if geometry == "cube":
        # cube rotate + pool: read q, k, v, write q^r, k^r, v in padded cube order; then the summary reads k, v
        pad = nB * 64 / cfg["N"]
        pre_bytes = (3 + 3 * pad + 2) * tensor_bytes
        pre_note = ("cube geometry: read q, k, v + write q^r, k^r, v in padded cube order (x%.3f) + the "
                    "summary's second read of k, v; algorithmic_bytes = one read of q, k, v" % pad)
    select_flops = 2.0 * cfg["B"] * cfg["H"] * nB * nB * 128
    secondary = {
        "prepass": {"bound": "hbm", "achieved_gbs": pre_bytes / (stage_ms["prepass"] * 1e-3) / 1e9,
                    "peak_gbs": hbm, "frac": pre_bytes / (stage_ms["prepass"] * 1e-3) / 1e9 / hbm,
                    "bytes": pre_bytes, "algorithmic_bytes": 3 * tensor_bytes, "note": pre_note},
        "select": {"bound": "fp32", "ms": stage_ms["select"], "flops": select_flops,
                   "achieved_tflops": select_flops / (stage_ms["select"] * 1e-3) / 1e12,
                   "note": "block scores (fp32 FMA) + per-row top-k + summary combine"},
        "apply_fuse": {"bound": "hbm",
                       "achieved_gbs": 3 * tensor_bytes / (stage_ms["apply_fuse"] * 1e-3) / 1e9, "peak_gbs": hbm,
                       "frac": 3 * tensor_bytes / (stage_ms["apply_fuse"] * 1e-3) / 1e9 / hbm,
                       "bytes": 3 * tensor_bytes, "note": "read q and O^s, write O"},
    }

    # ---- the token gate g = sigmoid(X w_g + b_g) from the block input X [B][N][H*128]
    # (an input of the layer step above; timed on its own)
    d_model = cfg["H"] * 128
    xg = inputs.make_gate_inputs(cfg["B"], cfg["N"], d_model, dtype=torch.bfloat16, device=dev, seed=7)
    gbuf = torch.empty((cfg["B"], cfg["N"]), dtype=torch.float32, device=dev)
    for _ in range(3):
        rola.gate(c, xg["X"], xg["w_g"], xg["b_g"], gbuf)
    torch.cuda.synchronize()
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0.record(stream)
    for _ in range(10):
        rola.gate(c, xg["X"], xg["w_g"], xg["b_g"], gbuf)
    g1.record(stream)
    torch.cuda.synchronize()
    gate_ms = g0.elapsed_time(g1) / 10
    gate_bytes = float(xg["X"].numel() * 2 + d_model * 2 + gbuf.numel() * 4)
    secondary["gate"] = {"bound": "hbm", "ms": gate_ms, "bytes": gate_bytes,
                         "achieved_gbs": gate_bytes / (gate_ms * 1e-3) / 1e9, "peak_gbs": hbm,
                         "frac": gate_bytes / (gate_ms * 1e-3) / 1e9 / hbm,
                         "note": f"X [B][N][{d_model}] bf16 read once ({xg['X'].numel() * 2 / 1e6:.0f} MB)"}
    del xg, gbuf

    # ---- the output projection Y = concat_h(O) W_o^T + b_o on the layer's output o (the block's
    # last step; a tcgen05 GEMM, B*N x d_model x H*128), timed on its own
    wo = (torch.randn((d_model, d_model), device=dev) / d_model ** 0.5).to(torch.bfloat16)
    bo = 0.1 * torch.randn((d_model,), device=dev)
    ybuf = torch.empty((cfg["B"], cfg["N"], d_model), dtype=torch.bfloat16, device=dev)
    for _ in range(3):
        rola.out_proj(c, o, wo, bo, ybuf, wsb)
    torch.cuda.synchronize()
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    p0.record(stream)
    for _ in range(10):
        rola.out_proj(c, o, wo, bo, ybuf, wsb)
    p1.record(stream)
    torch.cuda.synchronize()
    assert rola.get_device_status(wsb) == rola.ROLA_OK
    proj_ms = p0.elapsed_time(p1) / 10
    proj_flops = 2.0 * cfg["B"] * cfg["N"] * d_model * d_model
    secondary["out_proj"] = {"bound": "tensor", "ms": proj_ms, "flops": proj_flops,
                             "achieved_tflops": proj_flops / (proj_ms * 1e-3) / 1e12, "peak_tflops": peak,
                             "frac": proj_flops / (proj_ms * 1e-3) / 1e12 / peak,
                             "note": f"Y [B][N][{d_model}] = concat_h(O) W_o^T + b_o, bf16 in/out, fp32 accumulation; "
                                     "peak = measured bf16 burst"}
    del wo, bo, ybuf

    # ---- end to end through the public API with host buffers
    # Every step copies its inputs from pinned host memory and reads its output
    # back.  Serial: copy in, layer, copy out on one stream.  Pipelined (the
    # reported value): step i+1's inputs travel on a copy stream and step i's
    # output on another while step i's layer runs; two device buffer sets.
    e2e = None
    if not args.no_e2e:
        host = {k: (None if v is None else v.cpu().pin_memory()) for k, v in x.items()}
        o_host = [torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for _ in range(2)]
        dbuf = [{k: (None if v is None else torch.empty_like(v)) for k, v in x.items()} for _ in range(2)]
        obuf = [o, torch.empty_like(o)]
        h2d = sum(v.numel() * v.element_size() for v in host.values() if v is not None)
        d2h = o_host[0].numel() * o_host[0].element_size()
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

        def copy_in(b):
            for kk, v in host.items():
                if v is not None:
                    dbuf[b][kk].copy_(v, non_blocking=True)

        def layer(b):
            d = dbuf[b]
            rola.forward(c, d["q"], d["k"], d["v"], d["P_q"], d["P_k"], d["gate"], obuf[b], kv, wsb)

        def serial_steps(n):
            for _ in range(n):
                copy_in(0)
                layer(0)
                o_host[0].copy_(obuf[0], non_blocking=True)

        def pipelined_steps(n):
            loaded = [torch.cuda.Event() for _ in range(2)]
            done = [torch.cuda.Event() for _ in range(2)]
            read = [torch.cuda.Event() for _ in range(2)]
            s_in.wait_stream(stream)
            with torch.cuda.stream(s_in):
                copy_in(0)
                loaded[0].record(s_in)
            for i in range(n):
                b = i & 1
                if i + 1 < n:                                  # prefetch step i+1 into the other set
                    with torch.cuda.stream(s_in):
                        if i >= 1:
                            s_in.wait_event(done[b ^ 1])       # layer i-1 has finished reading it
                        copy_in(b ^ 1)
                        loaded[b ^ 1].record(s_in)
                stream.wait_event(loaded[b])
                if i >= 2:
                    stream.wait_event(read[b])                 # output i-2 has left the buffer
                layer(b)
                done[b].record(stream)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(done[b])
                    o_host[b].copy_(obuf[b], non_blocking=True)
                    read[b].record(s_out)
            stream.wait_stream(s_out)

        def timed(fn, n):
            fn(2)
            torch.cuda.synchronize()
            barrier(ws)
            a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn(n)
            z.record(stream)
            torch.cuda.synchronize()
            return reduce_max(a.elapsed_time(z) / n, ws)

        # the host link on its own: one step's inputs in and one output back, each timed alone
        torch.cuda.synchronize()
        l0, l1, l2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        with torch.cuda.stream(s_in):
            l0.record(s_in)
            copy_in(0)
            l1.record(s_in)
            o_host[0].copy_(obuf[0], non_blocking=True)
            l2.record(s_in)
        torch.cuda.synchronize()
        link = {"h2d_gbs": h2d / (l0.elapsed_time(l1) * 1e-3) / 1e9, "d2h_gbs": d2h / (l1.elapsed_time(l2) * 1e-3) / 1e9}
        ke = max(4, K)
        serial_ms = timed(serial_steps, max(2, K // 2))
        # three timed windows of ke pipelined steps; the median window is reported (the host link's
        # speed varied between processes on one box, so one window alone is a noisy sample)
        windows = [timed(pipelined_steps, ke) for _ in range(3)]
        e_ms = sorted(windows)[1]
        assert rola.get_device_status(wsb) == rola.ROLA_OK
        e2e = {"value": job_throughput(tokens, e_ms, ws), "unit": "tokens/s", "ms_per_step": e_ms,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": ke,
               "windows_ms_per_step": windows, "link": link,
               "mode": "pipelined: step i+1's host-to-device copies and step i's device-to-host read overlap "
                       "step i's layer on two copy streams; median of three timed windows",
               "serial": {"value": job_throughput(tokens, serial_ms, ws), "ms_per_step": serial_ms}}
        del dbuf, obuf

    # ---- dense comparator: the same kernels with every block kept
    dense = None
    if not args.no_dense:
        cd = rola.make_config(dict(cfg, keep=1.0))
        wsd = rola.workspace(cd, dev)
        kvd = torch.empty((cfg["B"], cfg["H"], rola.num_query_blocks(cd), nB), dtype=torch.int32, device=dev)
        rola.forward(cd, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], o, kvd, wsd)
        torch.cuda.synchronize()
        s3, t3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s3.record(stream)
        for _ in range(2):
            rola.forward(cd, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], o, kvd, wsd)
        t3.record(stream)
        torch.cuda.synchronize()
        d_ms = s3.elapsed_time(t3) / 2
        qsz = block_sizes(cfg, 128) if cfg.get("qblock", 0) == 128 else None
        flop_ratio = (sparse_flops_from_mask(kvd, block_sizes(cfg), qsizes=qsz) +
                      lowrank_flops(1, cfg["H"], cfg["N"], 128, cfg["r"])) / \
            (fl + lowrank_flops(1, cfg["H"], cfg["N"], 128, cfg["r"]))
        dense = {"dense_ms": d_ms, "speedup": d_ms / ms_step, "flop_ratio": flop_ratio,
                 "target_speedup": 0.85 * flop_ratio}
        del wsd, kvd

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu:
        cpu = cpu_oracle_estimate(cfg)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws, "steps": K, "warmup": args.warmup,
            "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": {"workload": cfg["name"], "B": cfg["B"], "H": cfg["H"], "N": cfg["N"],
                       "grid": [cfg["T"], cfg["Hh"], cfg["Ww"]], "block": 64, "keep": cfg["keep"],
                       "n_keep": nk, "r": cfg["r"], "d_h": 128, "lowrank_act": cfg.get("lowrank_act", "silu"),
                       "block_geometry": cfg.get("block_geometry", "flat"),
                       "query_block": cfg.get("qblock", 0) or 64,
                       "l2": "no flush: q, k, v are each larger than L2 (774 MB vs 129 MB)",
                       "parallelism": f"replica per GPU x{ws}"},
            "stage_ms": stage_ms,
            "step_ms": step_stats,
            "roofline": roofline,
            "roofline_other": secondary,
            "dense": dense,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": LAUNCHES_PER_FORWARD[geometry] * K,
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
