#!/usr/bin/env python
"""Benchmark of MoNe test-time learning on GB300 (one JSON line on stdout).

One step = one pass of the whole hot path over one synthetic context: reset the
fast weights to W_0, test-time learning of every layer's memory over all N/T
segments (prepass, phase A, phase B per segment, final renormalisation), then
the memory read (generate_kv) for a Q-token query.  Inputs are resident in HBM
when the timed region starts; the e2e figure repeats the step with the context
in pinned host memory (mone_ttl_context_host streams it over the host link inside
the timed region), the query copied in and the generated K/V copied back.

--impl reference times the fp64 CPU oracle (the comparison point: the paper ships
no implementation) on the host cores over a bounded sample of the same workload.

Multi-GPU (torchrun): every rank runs an independent replica of the workload
(independent contexts; no collective on the data path); value = all ranks'
tokens / max time over ranks, scaling "weak".
"""
from __future__ import annotations

import argparse
import csv
import hashlib
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

METRIC = "test-time-learning context tokens/sec at 128K (1 GB300); tensor-pipe util %"
UNIT = "tokens/s"
# datasheet figures, reported beside the measured peaks: HBM3e bandwidth and dense bf16 tensor rate
NOMINAL_HBM_GBS = 8000.0
L2_BYTES = 129 * 1024 * 1024   # GB300 L2; a working set above it is not served from L2
NOMINAL_BF16_TFLOPS = 2250.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="l16_d2048_128k")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=15.0, help="target CPU time of the oracle sample")
    p.add_argument("--n-tokens", type=int, default=0, help="override the context length (small profiling cases)")
    p.add_argument("--loss", default="neg_inner", choices=["neg_inner", "mse"],
                   help="per-token loss: Eq. 7 (the measured workload) or the squared-error variant")
    p.add_argument("--renorm-axis", default="rows", choices=["rows", "out"],
                   help="paper-mode renormalisation channels: rows of W1 and W2, or W1 rows and W2 columns")
    p.add_argument("--gate", default="linear", choices=["linear", "silu"], help="read gate: g_h or SiLU(g_h)")
    return p.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def fp32_alu_peak_tflops(dev):
    """FP32 FMA peak of the CUDA cores: SMs x 128 FP32 lanes x 2 flop x the maximum SM clock
    (the fp32 path's contractions run on them, not on the tensor cores)."""
    import torch
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mhz = float(json.load(f)["sm_max_mhz"])
    except Exception:
        mhz = 2070.0
    return sms * 128 * 2 * mhz * 1e6 / 1e12


# ------------------------------------------------------------------ algorithmic work per launch

def fast_params(wl):
    """Fast weights per chain: d_hid (d_in + d_out) for the MLP, 3 d_hid d_in for the SwiGLU heads."""
    return 3 * wl.d_hid * wl.d_in if wl.memory == "swiglu" else wl.d_hid * (wl.d_in + wl.d_out)


def flops_per_token(wl):
    """Algorithmic work of one token on one chain (forward + backward of the memory): the MLP's
    4 (d_in d_hid + d_hid d_out); the SwiGLU heads' 4 x 3 d_hid dh per head (two forward
    contractions, the backward one R, three gradients)."""
    if wl.memory == "swiglu":
        return 12 * wl.d_hid * wl.d_in
    return 4 * (wl.d_in * wl.d_hid + wl.d_hid * wl.d_out)


def kernel_work(wl, kind, chains=None):
    """(flops, bytes) of one launch of a phase kernel: one segment of `chains` chains
    (all of them by default; the library runs the chains of a call in two groups)."""
    C, T = (wl.chains if chains is None else chains), wl.seg_T
    di, dh, do = wl.d_in, wl.d_hid, wl.d_out
    params = fast_params(wl)
    flops = T * flops_per_token(wl) * C // 2
    act = T * (di + do) * 2            # U and Y tiles, bf16, read once
    grads = T * dh * 2 * (2 if wl.memory == "mlp" else 3 * wl.heads)  # phase A outputs, bf16
    if kind == "resident":
        # fp32 chains resident on chip: `chains` counts chain-segments; U and Y (fp32) stream
        # once, and W (and mu in paper mode) cross HBM once per launch (a window of segments)
        state = wl.chains * params * (8 + (8 if wl.mode == 1 else 0))
        return T * flops_per_token(wl) * C, C * T * (di + do) * 4 + state
    if kind == "phase_a":
        byts = C * (act + grads + params * 2)          # + bf16 weight operand read
    else:
        state = params * (4 + 4 + 2)                   # W fp32 read + write, bf16 copy write
        if wl.mode == 1:
            state += params * 8                        # momentum fp32 read + write
        byts = C * (act + grads + state)
    return flops, byts


def e2e_breakdown(context_bytes, gather_ms, gathers, gather_busy_ms, step_ms):
    """Where the end-to-end step's time goes, from one instrumented step: the library's host-input
    gathers (kernel kind "stage": `gathers` launches, `gather_ms` summed, `gather_busy_ms` the
    union of their intervals) moved `context_bytes` over the host link.  The achieved link rate,
    and the share of the step during which a gather was running, tell a slow link apart from a
    stalled pipeline (a step near the gathers' busy time is bound by the link)."""
    busy = gather_busy_ms if gather_busy_ms > 0 else gather_ms
    return {"h2d_gbs": context_bytes / (busy / 1000) / 1e9 if busy > 0 else None,
            "gathers_per_step": gathers,
            "gather_ms_mean": gather_ms / gathers if gathers else None,
            "gather_busy_ms_per_step": busy,
            "gather_share_of_step": busy / step_ms if step_ms > 0 else None}


def dominant_roofline(wl, dom, d, busy_ms, timed_segments, timed_ms, pk, alu_peak=None, traffic=None):
    """Roofline of the dominant kernel of the step.

    The work is the algorithmic work of the path: 2 T d_hid (d_in + d_out) flops per
    chain-segment for each phase kernel (half of the 4 (d_in d_hid + d_hid d_out) per token of
    forward plus backward).  On the bf16 path it is set against the tensor peak: the sustained
    one, since the kernel is timed inside a long step (`frac`), and the burst one beside it.
    `achieved` is one launch's work over the kernel's average launch duration; `busy` is the
    work of all timed launches over the union of their launch intervals on both streams (the
    two chain groups' launches overlap, so the average launch duration counts shared time
    twice).  Phase B also streams the fp32 state (W and mu read and written, the bf16 operand
    copy written): its bytes with that state are under `hbm`, against the HBM peak.  The fp32
    path's resident kernel runs on the CUDA cores: its flops are set against the FP32 FMA peak."""
    hbm, tf_burst, tf_sus, src = pk
    flops1, byts1 = kernel_work(wl, dom, d["chains_per_launch"])
    avg_s = d["avg_us"] * 1e-6
    flops_all, byts_all = kernel_work(wl, dom, wl.chains)
    if alu_peak:
        ach = flops1 / avg_s / 1e12
        roof = {"kernel": dom, "bound": "alu", "achieved": ach, "peak": alu_peak, "unit": "TFLOP/s",
                "frac": ach / alu_peak, "traffic": traffic,
                "peak_source": "FP32 FMA: SMs x 128 lanes x 2 flop x max SM clock"}
        if busy_ms > 0:
            b = flops_all * timed_segments / (busy_ms / 1000) / 1e12
            roof["busy"] = {"ms": busy_ms, "share_of_steps": busy_ms / timed_ms, "achieved": b,
                            "frac": b / alu_peak, "unit": "TFLOP/s"}
        return roof
    ach = flops1 / avg_s / 1e12
    roof = {"kernel": dom, "bound": "tensor", "achieved": ach, "peak": tf_sus, "unit": "TFLOP/s",
            "frac": ach / tf_sus, "frac_of_burst": ach / tf_burst, "traffic": traffic,
            "peak_source": f"{src} bf16_tflops_sustained (burst: bf16_tflops)",
            "work": "2 T d_hid (d_in + d_out) flops per chain-segment, algorithmic"}
    if busy_ms > 0:
        b = flops_all * timed_segments / (busy_ms / 1000) / 1e12
        roof["busy"] = {"ms": busy_ms, "share_of_steps": busy_ms / timed_ms, "achieved": b, "frac": b / tf_sus,
                        "frac_of_burst": b / tf_burst, "unit": "TFLOP/s"}
    if dom == "phase_b":
        g = byts1 / avg_s / 1e9
        roof["hbm"] = {"achieved": g, "peak": hbm, "unit": "GB/s", "frac": g / hbm,
                       "bytes_per_launch": byts1,
                       "bytes_note": "state-inclusive: W and mu read and written in fp32 and the bf16 operand "
                                     "copy written every segment (18 B per parameter), plus U, Y, dH, At"}
        if busy_ms > 0:
            gb = byts_all * timed_segments / (busy_ms / 1000) / 1e9
            roof["hbm"]["busy"] = {"achieved": gb, "frac": gb / hbm}
    if d["chains_per_launch"] < wl.chains:
        roof["note"] = ("launches of the two chain groups run concurrently on two streams; a launch's "
                        "duration includes the SMs and HBM bandwidth the other group's kernels take, "
                        "so two overlapping launches each count the shared time; 'busy' divides the "
                        "kernel's algorithmic work over the timed steps by the union of its launch "
                        "intervals instead")
    return roof


def kernel_source_sha(text, kind):
    """sha256[:16] of one kernel's section of ttl_tc.cu (phase B: from its section banner to
    make_args), so that the recorded counters stay valid while that kernel's source is unchanged."""
    if kind != "phase_b":
        return None
    i = text.index("// ------------------------------------------------------------------ phase B")
    j = text.index("TcArgs make_args(")
    return hashlib.sha256(text[i:j].encode()).hexdigest()[:16]


def shape_key(wl):
    """The per-chain shape a DRAM-traffic record holds for (widths, segment, memory form, mode, loss)."""
    return (f"{wl.d_in}x{wl.d_hid}x{wl.d_out}:T{wl.seg_T}:{wl.memory}:{'paper' if wl.mode == 1 else 'plain'}:"
            f"{wl.loss}")


def ncu_traffic(kind, chains, wl):
    """DRAM bytes per launch of `chains` chains from the committed ncu summary (scaled from the
    captured launch's chain count), if the kernel source is unchanged and the record was taken
    on this per-chain shape."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    src = os.path.join(ROOT, "paper_2608_17616_gb300", "csrc", "ttl_tc.cu")
    try:
        sha = kernel_source_sha(open(src).read(), kind)
        for line in open(path):
            if line.lstrip().startswith("#"):
                continue
            parts = dict(kv.split("=", 1) for kv in line.split() if "=" in kv)
            if (parts.get("kernel") == kind and parts.get("source_sha") == sha
                    and parts.get("shape") == shape_key(wl)):
                cap = float(parts.get("chains", chains))
                note = parts.get("scaled_from", "")
                if abs(cap - chains) > 1e-9:
                    note = f"{note}; scaled from a {cap:g}-chain launch to {chains:g} chains"
                return float(parts["bytes_per_launch"]) * chains / cap, note
    except Exception:
        pass
    return None, ""


# ------------------------------------------------------------------ clocks

class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.p = None
        self.idx = gpu_index
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        time.sleep(0.3)
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.flush()
        rows = []
        with open(self.f.name) as fh:
            for r in csv.reader(fh):
                if len(r) >= 9:
                    rows.append([x.strip() for x in r])
        os.unlink(self.f.name)
        if not rows:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1])]
        mx = [num(r[2]) for r in rows if num(r[2])]
        pw = [num(r[3]) for r in rows if num(r[3])]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        loaded = [s for s, p in zip(sm, pw) if p is not None and p > 0.35 * max(pw)] if pw else sm
        return {"sm_mhz": statistics.median(loaded or sm), "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


# ------------------------------------------------------------------ oracle timing (CPU baseline / reference arm)

_ORACLE_INPUTS = {}


def oracle_sample(wl, seconds, chain=0):
    """Time the fp64 oracle on chain `chain`, segment after segment (continuing the chain),
    until ~`seconds` have elapsed or the context ends.  The inputs are drawn once (a prefix
    sized from a two-segment calibration) and kept for later samples of the same run.

    Returns (tokens_per_s in whole-context tokens, sample description, cores, seconds)."""
    import numpy as np

    import oracle as O
    import workloads as wk
    T = wl.seg_T
    W1all, W2all = wk.initial_weights(wl, "cpu")
    W1, W2 = W1all[chain], W2all[chain]
    meta = O.Meta.from_torch(wk.meta_params(wl, "cpu"), chain) if wl.mode == wk.PAPER else None
    hp = O.Hyper(mode=wl.mode, lr=wl.lr, loss=wl.loss, memory=wl.memory, n_heads=wl.heads,
                 renorm_axis=wl.renorm_axis, gate_act=wl.gate_act)

    def init():
        if wl.memory == "swiglu":
            return O.init_state(Win=O.f64(W1[:, :wl.d_hid]), Wg=O.f64(W1[:, wl.d_hid:]), Wout=O.f64(W2))
        return O.init_state(W1=O.f64(W1), W2=O.f64(W2))

    def inputs(n_seg):
        key = (wl.name, chain)
        have = _ORACLE_INPUTS.get(key)
        if have is None or have[0].shape[0] < n_seg * T:
            x, k, v = wk.chain_inputs(wl, chain, "cpu", n_seg * T)
            have = (x, torch_cat(k, v))
            _ORACLE_INPUTS[key] = have
        return have

    def torch_cat(k, v):
        import torch
        return torch.cat([k, v], dim=1)

    # calibration: two segments after one of warm-up
    x, y = inputs(min(3, wl.S))
    st = init()
    cal = min(3, wl.S)
    t_cal = 0.0
    for i in range(cal):
        Xs, Ys = O.f64(x[i * T:(i + 1) * T]), O.f64(y[i * T:(i + 1) * T])
        t0 = time.perf_counter()
        st, _ = O.ttl_context(st, Xs, Ys, T, hp, meta)
        if i > 0 or cal == 1:
            t_cal += time.perf_counter() - t0
    per_seg = t_cal / max(1, cal - 1)
    n_need = int(min(wl.S, max(1, 1.5 * seconds / max(per_seg, 1e-6))))
    x, y = inputs(n_need)
    st = init()
    n_seg = 0
    dt = 0.0
    while n_seg < n_need and dt < seconds:
        Xs = O.f64(x[n_seg * T:(n_seg + 1) * T])
        Ys = O.f64(y[n_seg * T:(n_seg + 1) * T])
        t0 = time.perf_counter()
        st, _ = O.ttl_context(st, Xs, Ys, T, hp, meta)
        dt += time.perf_counter() - t0
        n_seg += 1
    chain_tokens_per_s = n_seg * T / dt
    # a context token needs one chain-token of work in every layer
    tok_s = chain_tokens_per_s / wl.n_layers
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", "0") or 0) or os.cpu_count()
    sample = (f"oracle (fp64 NumPy) on chain {chain} of {wl.name}: {n_seg} segment(s) x T={T} = {n_seg * T} tokens "
              f"of one layer in {dt:.2f} s (the chain continued segment by segment); scaled to whole-context "
              f"tokens by 1/{wl.n_layers} layers")
    return tok_s, sample, cores, dt


# ------------------------------------------------------------------ arms

def max_over_ranks(x: float, device="cpu") -> float:
    """The largest value of x over all ranks (x itself without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(ms_local: float, tokens_per_rank: int, world: int, device="cpu"):
    """(ms per step, whole-job tokens/s): every rank's tokens over the slowest rank's time."""
    ms = max_over_ranks(ms_local, device)
    return ms, world * tokens_per_rank / (ms / 1000.0)


def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def run_reference(args, wl):
    ws, rank, _ = dist_setup()
    if rank != 0:
        return
    rates = []
    sample = ""
    cores = os.cpu_count()
    per_step = max(2.0, min(20.0, 150.0 / max(1, args.steps + args.warmup)))
    t_all = []
    for i in range(args.warmup + args.steps):
        r, sample, cores, dt = oracle_sample(wl, per_step)
        if i >= args.warmup:
            rates.append(r)
            t_all.append(dt)
    val = statistics.median(rates)
    line = {"metric": METRIC, "value": val, "unit": UNIT, "impl": "reference", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * statistics.median(t_all),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(wl),
            "cpu_baseline": {"value": val, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def config_of(wl):
    return {"workload": wl.name, "n_ctx": wl.n_ctx, "n_layers": wl.n_layers, "chains": wl.chains,
            "N": wl.N, "seg_T": wl.seg_T, "d_in": wl.d_in, "d_hid": wl.d_hid, "d_out": wl.d_out, "Q": wl.Q,
            "mode": "paper" if wl.mode == 1 else "plain", "loss": wl.loss, "memory": wl.memory, "heads": wl.heads,
            "renorm_axis": wl.renorm_axis, "gate": wl.gate_act,
            "masters": "fp32", "operands": wl.dtype,
            "l2": "inputs larger than L2 (no flush needed)"}


def run_ours(args, wl):
    import torch

    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_17616_gb300 as mone
    import workloads as wk

    dev = f"cuda:{local}"
    W1_0, W2_0 = wk.initial_weights(wl, dev)
    meta = wk.meta_params(wl, dev) if wl.mode == wk.PAPER else None
    X, K, V = wk.all_inputs(wl, dev)
    Xq = wk.query_inputs(wl, dev)
    mu0_1 = torch.zeros_like(W1_0) if wl.mode == wk.PAPER else None
    mu0_2 = torch.zeros_like(W2_0) if wl.mode == wk.PAPER else None
    Kout = torch.empty(wl.n_ctx, wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim, dtype=X.dtype, device=dev)
    Vout = torch.empty_like(Kout)
    strides = mone.kv_strides(wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim)
    cfg = mone.make_config(wl.n_ctx, wl.n_layers, wl.d_in, wl.d_hid, wl.d_out, wl.n_kv_heads, wl.head_dim, wl.seg_T,
                           mone.MONE_FP32 if wl.dtype == "f32" else mone.MONE_BF16, wl.mode, wl.lr,
                           loss=mone.MONE_LOSS_MSE if wl.loss == "mse" else mone.MONE_LOSS_DOT,
                           memory=mone.MONE_MEM_SWIGLU if wl.memory == "swiglu" else mone.MONE_MEM_MLP,
                           mem_heads=wl.heads,
                           renorm_axis=mone.MONE_RENORM_OUT if wl.renorm_axis == "out" else mone.MONE_RENORM_ROWS,
                           gate_act=mone.MONE_GATE_SILU if wl.gate_act == "silu" else mone.MONE_GATE_LINEAR)
    h = mone.mone_mem_init(cfg, W1_0, W2_0, meta)
    stream = torch.cuda.current_stream()

    def step(x=X, k=K, v=V, xq=Xq):
        mone.mone_mem_write_state(h, W1_0, W2_0, mu0_1, mu0_2)
        mone.mone_ttl_context(h, x, k, v, wl.N)
        mone.mone_mem_generate_kv(h, xq, wl.Q, Kout, Vout, strides)

    def barrier():
        if ws > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(args.warmup):
        step()
    mone.mone_mem_sync(h)

    clocks = Clocks(local)
    mone.mone_mem_set_timing(h, True)
    n0 = mone.mone_mem_launch_count(h)
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = mone.mone_mem_launch_count(h) - n0
    ms = e0.elapsed_time(e1) / args.steps
    timed_segments = args.steps * ((wl.N + wl.seg_T - 1) // wl.seg_T)
    ktimes = {name: mone.mone_mem_kernel_time(h, i) for i, name in enumerate(mone.KERNEL_KINDS)}
    kbusy = {name: mone.mone_mem_kernel_busy(h, i) for i, name in enumerate(mone.KERNEL_KINDS)}
    mone.mone_mem_set_timing(h, False)
    clk = clocks.stop()
    mone.mone_mem_sync(h)
    tokens_per_step = wl.n_ctx * wl.N
    ms, value = job_rate(ms, tokens_per_step, ws, dev)

    # ---- end to end through the public calls with host buffers: the context is handed to the
    # library in pinned host memory (mone_ttl_context_host), which gathers chunks of whole segments
    # into its device windows while it learns the previous chunk; then the query is copied in, read,
    # and the memory K/V are copied back.
    e2e = None
    if not args.no_e2e:
        hX = torch.empty(X.shape, dtype=X.dtype, pin_memory=True)
        hK = torch.empty(K.shape, dtype=K.dtype, pin_memory=True)
        hV = torch.empty(V.shape, dtype=V.dtype, pin_memory=True)
        hX.copy_(X)
        hK.copy_(K)
        hV.copy_(V)
        hXq = torch.empty(Xq.shape, dtype=Xq.dtype, pin_memory=True)
        hXq.copy_(Xq)
        hKo = torch.empty(Kout.shape, dtype=Kout.dtype, pin_memory=True)
        hVo = torch.empty(Vout.shape, dtype=Vout.dtype, pin_memory=True)
        dXq = torch.empty_like(Xq)

        def e2e_step():
            mone.mone_mem_write_state(h, W1_0, W2_0, mu0_1, mu0_2)
            mone.mone_ttl_context_host(h, hX, hK, hV, wl.N)
            dXq.copy_(hXq, non_blocking=True)
            mone.mone_mem_generate_kv(h, dXq, wl.Q, Kout, Vout, strides)
            hKo.copy_(Kout, non_blocking=True)
            hVo.copy_(Vout, non_blocking=True)

        n_e2e = max(1, min(args.steps, 5))
        e2e_step()  # first call: the library sizes its staging windows
        torch.cuda.synchronize()
        barrier()
        e0.record(stream)
        for _ in range(n_e2e):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ms_e2e, _ = job_rate(e0.elapsed_time(e1) / n_e2e, tokens_per_step, ws, dev)
        h2d = sum(t.numel() * t.element_size() for t in (hX, hK, hV, hXq))
        d2h = sum(t.numel() * t.element_size() for t in (hKo, hVo))
        # one more step with the library's per-kernel timing on, for the breakdown (not timed above)
        mone.mone_mem_set_timing(h, True)
        e2e_step()
        st_ms, st_n = mone.mone_mem_kernel_time(h, mone.KERNEL_KINDS.index("stage"))
        st_busy = mone.mone_mem_kernel_busy(h, mone.KERNEL_KINDS.index("stage"))
        mone.mone_mem_set_timing(h, False)
        mone.mone_mem_sync(h)
        e2e = {"value": ws * tokens_per_step / (ms_e2e / 1000.0), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e, "api": "mone_ttl_context_host"}
        e2e.update(e2e_breakdown(h2d - hXq.numel() * hXq.element_size(), st_ms, st_n, st_busy, ms_e2e))

    # ---- consumer attention of the read (Eq. 5): the query's tokens over [memory tokens || their own
    # keys], timed on its own (it is not part of the test-time-learning step).  The memory tokens are
    # this step's read (Q of them); the query tokens' own Q, K, V are synthetic; 2 query heads per
    # key/value head.
    attn = None
    if ws == 1 or rank == 0:
        n_q, Lq, n_mem = 2 * wl.n_kv_heads, wl.Q, wl.Q
        ga = torch.Generator(device=dev).manual_seed(1234)
        cache = (wl.n_ctx, wl.n_layers, wl.n_kv_heads, n_mem + Lq, wl.head_dim)
        qshape = (wl.n_ctx, wl.n_layers, n_q, Lq, wl.head_dim)
        # enough independent input sets that one pass over them exceeds L2: each call reads
        # inputs last touched a full pass earlier
        one = (2 * math.prod(cache) + 2 * math.prod(qshape)) * X.element_size()
        n_sets = max(2, -(-L2_BYTES // one) + 1)
        sets = []
        for _ in range(n_sets):
            Kc = torch.randn(*cache, generator=ga, device=dev).to(X.dtype)
            Vc = torch.randn(*cache, generator=ga, device=dev).to(X.dtype)
            mone.mone_mem_generate_kv(h, Xq, wl.Q, Kc, Vc, Kc.stride()[:4])
            Qa = torch.randn(*qshape, generator=ga, device=dev).to(X.dtype)
            sets.append((Qa, Kc, Vc, torch.empty_like(Qa)))

        def attend_all():
            for Qa, Kc, Vc, Oa in sets:
                mone.mone_attention(h, Qa, n_q, Lq, Kc, Vc, Kc.stride()[:4], n_mem, Oa)

        for _ in range(3):
            attend_all()
        torch.cuda.synchronize()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        # eager: one library call per set from Python, back to back (includes the host's call rate)
        a0.record(stream)
        attend_all()
        a1.record(stream)
        torch.cuda.synchronize()
        us_eager = 1000 * a0.elapsed_time(a1) / n_sets
        # device time: the same calls captured once in a CUDA graph and replayed
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            attend_all()
        graph.replay()
        torch.cuda.synchronize()
        a0.record(stream)
        graph.replay()
        a1.record(stream)
        torch.cuda.synchronize()
        mone.mone_mem_sync(h)
        us = 1000 * a0.elapsed_time(a1) / n_sets
        del graph
        Qa, Kc, Vc, Oa = sets[0]
        byts = (Kc.numel() + Vc.numel() + Qa.numel() + Oa.numel()) * Qa.element_size()
        # causal over the query tokens: token i sees n_mem + i + 1 keys
        flops = 4 * wl.chains * n_q * wl.head_dim * (Lq * n_mem + Lq * (Lq + 1) // 2)
        attn = {"us": us, "us_eager": us_eager, "timing": f"CUDA graph of {n_sets} calls on distinct inputs "
                f"({n_sets * byts / 1e6:.0f} MB, more than L2)", "n_q_heads": n_q, "Lq": Lq, "n_mem": n_mem,
                "bytes": byts, "gbs": byts / (us * 1e-6) / 1e9, "tflops": flops / (us * 1e-6) / 1e12}
        del sets

    # ---- roofline of the dominant kernel
    hbm, tf_burst, tf_sus, peak_src = peaks()
    kern = {}
    for name in ("phase_a", "phase_b", "resident"):
        tot, n = ktimes[name]
        if n == 0:
            continue
        avg_ms = tot / n
        # chains per launch, from the launches the library made for the timed steps
        chains = wl.chains * timed_segments / n
        flops, byts = kernel_work(wl, name, chains)
        kern[name] = {"chains_per_launch": chains,
                      "share": tot / max(1e-9, sum(v[0] for v in ktimes.values())), "avg_us": 1000 * avg_ms,
                      "launches": n, "tflops": flops / (avg_ms / 1000) / 1e12,
                      "gbs": byts / (avg_ms / 1000) / 1e9}
    dom = max(kern, key=lambda k: kern[k]["share"])
    d = kern[dom]
    traffic, traffic_note = ncu_traffic(dom, d["chains_per_launch"], wl)
    alu_peak = fp32_alu_peak_tflops(dev) if wl.dtype == "f32" else None
    roof = dominant_roofline(wl, dom, d, kbusy.get(dom, 0.0), timed_segments, ms * args.steps,
                             (hbm, tf_burst, tf_sus, peak_src), alu_peak, traffic)
    if traffic_note.strip("; "):
        roof["traffic_note"] = traffic_note.strip("; ")
    # the memory read: latency of one generate_kv call and its weight-streaming rate
    gkv = None
    t_read, n_read = ktimes["read"]
    if n_read:
        us = 1000 * t_read / n_read
        el = 2 if wl.dtype == "bf16" else 4
        # weights streamed once: the bf16 operand copy on the bf16 path, the fp32 masters on the fp32 path
        byts = wl.chains * (fast_params(wl) * el + wl.Q * (wl.d_in + wl.d_out) * el)
        gkv = {"us": us, "bytes": byts, "gbs": byts / (us * 1e-6) / 1e9, "frac_of_hbm": byts / (us * 1e-6) / 1e9 / hbm,
               "Q": wl.Q}
    # the whole step against HBM: algorithmic bytes of every kernel of the step / step time
    S = (wl.N + wl.seg_T - 1) // wl.seg_T
    if "resident" in kern:  # one launch per input window, each streaming its segments
        n_win = max(1, round(ktimes["resident"][1] / args.steps))
        step_bytes = n_win * kernel_work(wl, "resident", wl.chains * S / n_win)[1]
    else:
        step_bytes = S * (kernel_work(wl, "phase_a")[1] + kernel_work(wl, "phase_b")[1])
    if wl.mode == 1:
        step_bytes += wl.chains * wl.N * wl.d_in * 2 * (2 if wl.dtype == "bf16" else 4)  # input transform: read X, write U
    step_roof = {"bytes_per_step": step_bytes, "achieved": step_bytes / (ms / 1000) / 1e9, "peak": hbm,
                 "unit": "GB/s", "frac": step_bytes / (ms / 1000) / 1e9 / hbm,
                 "frac_of_nominal_8000": step_bytes / (ms / 1000) / 1e9 / NOMINAL_HBM_GBS}
    total_flops = flops_per_token(wl) * wl.N * wl.chains
    tensor_util = total_flops / (ms / 1000) / 1e12 / tf_burst

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        r, sample, cores, _ = oracle_sample(wl, args.cpu_seconds)
        cpu = {"value": r, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
                "config": config_of(wl), "e2e": e2e, "gpu_launches": launches, "roofline": roof,
                "cpu_baseline": cpu, "clocks": clk,
                "tensor_util_of_burst_peak": tensor_util,
                "tensor_util_of_nominal_2250": tensor_util * tf_burst / NOMINAL_BF16_TFLOPS,
                "step_roofline": step_roof, "generate_kv": gkv,
                "consumer_attention": attn,
                "kernels": kern}
        print(json.dumps(line), flush=True)
    mone.mone_mem_free(h)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def main():
    args = parse()
    import workloads as wk
    wl = wk.WORKLOADS[args.workload]
    if args.n_tokens:
        wl = wl.replace(N=args.n_tokens)
    if args.loss != "neg_inner":
        wl = wl.replace(loss=args.loss)
    if args.renorm_axis != "rows" or args.gate != "linear":
        wl = wl.replace(renorm_axis=args.renorm_axis, gate_act=args.gate)
    if args.impl == "reference":
        run_reference(args, wl)
    else:
        run_ours(args, wl)


if __name__ == "__main__":
    main()
