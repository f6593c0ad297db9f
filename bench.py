"""Benchmark of the CCQ hot path on GB300.

One step = one CCQ chunkwise forward over the whole workload batch (one call
of ccq_gla_fwd / ccq_gdn_fwd, or one ccq_decode_step), inputs resident in HBM;
for the fwd+bwd workload one step is a training step of the layer: the
forward that saves checkpoints (ccq_gla_fwd_save) then ccq_gla_bwd.
The default workload is CCQ-GLA forward, bf16, B=8, H=16, T=4096,
Dk=Dv=128, chunk 64 (the metric's configuration).  Prints ONE JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   (the fp64 CPU oracle on host cores)

Multi-GPU (torchrun, one rank per GPU): every rank runs its own copy of the
workload (independent sequences, no data-path collective); value is the
total tokens of all ranks / the max over ranks of the timed region.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "CCQ chunked fwd tokens/s at T=4K,d=128 bf16; % of roofline (tensor/HBM)"
METRIC_FWDBWD = "CCQ-GLA chunked fwd+bwd tokens/s at T=4K,d=128 bf16; % of roofline (HBM)"
METRIC_GDN_FWDBWD = "CCQ-GDN chunked fwd+bwd tokens/s at T=4K,d=128 bf16; % of roofline (HBM)"
METRICS = {"glabwd": METRIC_FWDBWD, "gdnbwd": METRIC_GDN_FWDBWD}
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")

# Workloads: name -> (backbone, B, H, T, D, kernel name, description)
WORKLOADS = {
    "gla_bf16_4k": ("gla", 8, 16, 4096, 128),
    "gdn_bf16_4k": ("gdn", 8, 16, 4096, 128),
    "gla_bf16_20k": ("gla", 1, 16, 20480, 128),
    "gdn_bf16_20k": ("gdn", 1, 16, 20480, 128),
    "decode_b256": ("decode", 256, 16, 1, 128),
    "gla_bf16_4k_fwdbwd": ("glabwd", 4, 16, 4096, 128),
    "gdn_bf16_4k_fwdbwd": ("gdnbwd", 4, 16, 4096, 128),
    # packed variable-length sequences: B sequences of 100-4000 tokens (VARLEN_SEED), one launch
    "gla_bf16_varlen64": ("glavl", 64, 16, 0, 128),
    "gdn_bf16_varlen64": ("gdnvl", 64, 16, 0, 128),
}
VARLEN_SEED = 77


def varlen_lengths(n):
    """The sequence lengths of a packed workload: n draws from 100..4000 tokens."""
    import numpy as np
    return np.random.default_rng(VARLEN_SEED).integers(100, 4001, size=n).tolist()
KERNEL_SOURCES = {"gla": "ccq_gla_chunk.cu", "gdn": "ccq_gdn_chunk.cu", "decode": "ccq_recurrent.cu",
                  "glavl": "ccq_gla_chunk.cu", "gdnvl": "ccq_gdn_chunk.cu",
                  "glabwd": "ccq_gla_bwd.cu", "gdnbwd": ("ccq_gdn_bwd_kernels.cuh", "ccq_gdn_bwd_tc.cuh")}
KERNEL_NAMES = {"gla": "gla_chunk_kernel", "gdn": "gdn_wy_kernel + gdn_chunk_kernel",
                "glavl": "gla_chunk_kernel (packed sequences)", "gdnvl": "gdn_wy_kernel + gdn_chunk_kernel (packed sequences)",
                "decode": "decode_kernel",
                "glabwd": "whole step: forward (saving checkpoints) + gla_bwd_q_kernel + gla_bwd_state_kernel"
                          " + gla_bwd_kv_kernel",
                "gdnbwd": "whole step: forward (gdn_wy_kernel + gdn_chunk_kernel), the backward's forward recompute,"
                          " gdn_bwd_local_kernel + gdn_bwd_state_tc_kernel + gdn_bwd_suffix_kernel + gdn_bwd_kv_kernel"}


def gla_segments(B, H, T, sms):
    """Segments per sequence the library's default split picks (ccq_capi.cu)."""
    nc = (T + 63) // 64
    ns = sms // (B * H) if B * H * 2 <= sms else 1
    ns = max(1, min(ns, nc // 8, nc))
    per = (nc + ns - 1) // ns
    return (nc + per - 1) // per


def launches_per_step(kind, B, H, T, sms):
    """Kernel launches of one step: the segmented GLA forward is three kernels, the
    Gated DeltaNet forward two (WY, chunk) or four when segmented, the backward three,
    and every call that returns the position count adds the one-thread-per-row count
    update."""
    if kind in ("glavl", "gdnvl"):  # one launch (two for GDN: WY, chunk) plus the count update
        return 2 if kind == "glavl" else 3
    split = gla_segments(B, H, T, sms) > 1
    fwd = 3 if split else 1
    gdn = 4 if split else 2
    # the Gated DeltaNet training step runs the forward twice (the step's forward, then the
    # backward's recompute of the forward's per-chunk quantities) and four backward kernels
    return {"gla": fwd + 1, "gdn": gdn + 1, "decode": 1 + 1, "glabwd": fwd + 1 + 3, "gdnbwd": 2 * gdn + 1 + 4}[kind]


def algorithmic_bytes(kind, B, H, T, D):
    """Bytes one launch must move at minimum: every input read once, o written
    once, final fp32 states written once (initial states are zero / absent
    except for decode, whose cache is read and written)."""
    if kind in ("glavl", "gdnvl"):  # B sequences, T = the packed length
        per = algorithmic_bytes(kind[:3], 1, H, T, D) - H * (2 * D * D + D) * 4 - 8
        return per + B * (H * (2 * D * D + D) * 4 + 8)
    tok = B * T * H
    if kind == "glabwd":
        # forward: q, k, v, gk, lambda in, o out, final states out; backward:
        # q, k, v, gk, lambda, dout in, dq, dk, dv, dgk, dlambda and the three
        # initial-state gradients out (each pass reads its own inputs once)
        fwd = algorithmic_bytes("gla", B, H, T, D)
        bwd = tok * D * 2 * 5 + tok * 4 + tok * D * 2 * 4 + tok * 4 + B * H * (2 * D * D + D) * 4
        return fwd + bwd
    if kind == "gdnbwd":
        # forward as gdn; backward: q, k, v, dout (bf16) and g, beta, lambda (fp32) in, dq, dk, dv
        # (bf16) and dg, dbeta, dlambda (fp32) out, the three initial-state gradients out
        fwd = algorithmic_bytes("gdn", B, H, T, D)
        bwd = tok * D * 2 * 4 + tok * 4 * 3 + tok * D * 2 * 3 + tok * 4 * 3 + B * H * (2 * D * D + D) * 4
        return fwd + bwd
    if kind == "gla":
        return tok * D * 2 * 4 + tok * D * 2 + tok * 4 + B * H * (2 * D * D + D) * 4 + B * 8
    if kind == "gdn":
        return tok * D * 2 * 3 + tok * D * 2 + tok * 4 * 3 + B * H * (2 * D * D + D) * 4 + B * 8
    # decode: q, k, v, gate (bf16) + lambda in, o out, cache (S, C, m) read and written
    return tok * D * 2 * 4 + tok * 4 + tok * D * 2 + 2 * B * H * (2 * D * D + D) * 4 + 2 * B * 8


def algorithmic_flops(kind, B, H, T, D, C=64):
    """Dense tile FLOPs of the chunkwise algorithm (Algorithm 1 products)."""
    if kind in ("glavl", "gdnvl"):
        return sum(algorithmic_flops(kind[:3], 1, H, n, D, C) for n in varlen_lengths(B))
    nc = (T + C - 1) // C
    # GLA: four C x D x D products (Qbar S^K, Qg S, Ku^T V, Kbar^T Kbar) and four
    # C x C x D products (Qbar Kbar^T, W' Kbar, Qg Kg^T, A V), 2 FLOP per MAC.
    # GLA backward (ccq_gla_bwd.cu), its tcgen05 products per chunk (M x N x K):
    # q kernel: C x C x D (Sc, T1, T3), C x D x D (Zi, Dq, u, two for dkc),
    # C x D x C (W2 Kbar, P1 Kd, W2^T DZ, W3 Kbar, W3^T Qbar), D x D x C (DC),
    # D x C x C twice (Dm); kv kernel: C x C x D (T1, SA), C x D x D (dkw, dv),
    # D x D x C (dS), C x D x C (P1^T QG, SA dO).
    bwd = 2 * (3 * C * C * D + 5 * C * D * D + 5 * C * D * C + D * D * C + 2 * D * C * C
               + 2 * C * C * D + 2 * C * D * D + D * D * C + 2 * C * D * C)
    # Gated DeltaNet backward (ccq_gdn_bwd_kernels.cuh), its products per chunk summed over the
    # prep, state, local and kv passes: fifteen C x D x D, twenty-two C x C x D, two C x C x C.
    gbwd = 2 * (15 * C * D * D + 22 * C * C * D + 2 * C * C * C)
    per_chunk = {"gla": 8 * C * D * D + 8 * C * C * D,
                 "gdn": 10 * C * D * D + 12 * C * C * D,
                 "glabwd": 8 * C * D * D + 8 * C * C * D + bwd,
                 "gdnbwd": 10 * C * D * D + 12 * C * C * D + gbwd}.get(kind)
    if per_chunk is None:
        return B * H * 8 * D * D
    return B * H * nc * per_chunk


# The kernels of one step of each workload and the source file of each kernel.
STEP_KERNELS = {
    "gla_bf16_4k": ["gla_chunk_kernel"],
    "gdn_bf16_4k": ["gdn_wy_kernel", "gdn_chunk_kernel"],
    "gla_bf16_20k": ["gla_segment_state_kernel", "gla_segment_combine_kernel", "gla_chunk_kernel"],
    "gdn_bf16_20k": ["gdn_wy_kernel", "gdn_segment_state_kernel", "gdn_segment_combine_kernel",
                     "gdn_chunk_kernel"],
    "decode_b256": ["decode_kernel"],
    "gla_bf16_4k_fwdbwd": ["gla_segment_state_kernel", "gla_segment_combine_kernel", "gla_chunk_kernel",
                           "gla_bwd_q_kernel", "gla_bwd_state_kernel", "gla_bwd_kv_kernel"],
    # (the forward kernels run twice: the forward itself, then the backward's recompute of the
    # forward's per-chunk quantities; segment-parallel at B = 4, H = 16)
    "gdn_bf16_4k_fwdbwd": ["gdn_segment_state_kernel", "gdn_segment_combine_kernel", "gdn_wy_kernel",
                           "gdn_chunk_kernel", "gdn_bwd_local_kernel", "gdn_bwd_state_tc_kernel",
                           "gdn_bwd_suffix_kernel", "gdn_bwd_kv_kernel"],
    "gla_bf16_varlen64": ["gla_chunk_kernel"],
    "gdn_bf16_varlen64": ["gdn_wy_kernel", "gdn_chunk_kernel"],
}
# (each step also runs the one-thread-per-row position update: 8 bytes per batch row, not counted)
KERNEL_FILES = {"gla_chunk_kernel": "ccq_gla_chunk.cu", "gla_segment_state_kernel": "ccq_gla_segment.cu",
                "gla_segment_combine_kernel": "ccq_gla_segment.cu", "gdn_wy_kernel": "ccq_gdn_chunk.cu",
                "gdn_chunk_kernel": "ccq_gdn_chunk.cu",
                "gdn_segment_state_kernel": "ccq_gdn_segment.cu", "gdn_segment_combine_kernel": "ccq_gdn_segment.cu", "recurrent": "ccq_recurrent.cu",
                "decode_kernel": "ccq_recurrent.cu", "gla_bwd_state_kernel": "ccq_gla_bwd.cu",
                "gla_bwd_q_kernel": "ccq_gla_bwd.cu", "gla_bwd_kv_kernel": "ccq_gla_bwd.cu",
                "gdn_bwd_state_tc_kernel": "ccq_gdn_bwd_state_tc.cu",
                **{f"gdn_bwd_{n}_kernel": "ccq_gdn_bwd_kernels.cuh"
                   for n in ("prep", "prefix", "fstate", "dstate", "suffix")},
                **{f"gdn_bwd_{n}_kernel": ("ccq_gdn_bwd_kernels.cuh", "ccq_gdn_bwd_tc.cuh") for n in ("local", "kv")}}


SHARED_DEVICE_SOURCES = ("sm100_ptx.cuh", "ccq_internal.h")  # inlined into every kernel


def source_sha(fname):
    """Hash of a kernel's source file (or files) and the device headers every kernel inlines."""
    h = hashlib.sha256()
    for f in (fname if isinstance(fname, tuple) else (fname,)) + SHARED_DEVICE_SOURCES:
        with open(os.path.join(ROOT, "paper_2606_01294_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def kernel_sha(kind):
    return source_sha(KERNEL_SOURCES[kind])


def measured_traffic(kind, workload):
    """DRAM bytes of one step (summed over its kernels) from the committed ncu
    captures, if every kernel of the step was captured on its current source;
    else None."""
    try:
        with open(TRAFFIC_FILE) as f:
            t = json.load(f).get(workload, {})
        total = 0
        for k in STEP_KERNELS[workload]:
            e = t.get(k)
            if not e or e.get("source_sha") != source_sha(KERNEL_FILES[k]):
                return None
            total += e["dram_bytes_per_launch"] * e.get("launches_per_step", 1)
        return total
    except (OSError, ValueError, KeyError):
        return None


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []
        self.window = None  # (start, end) wall-clock seconds of the timed region

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
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

    def summary(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        rows = []
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append((ts, float(parts[1]), float(parts[2]),
                             [n for n, v in zip(names, parts[5:9]) if v.lower() == "active"]))
            except (ValueError, IndexError):
                continue
        inside = rows
        where = "timed region"
        if self.window:
            inside = [r for r in rows if self.window[0] - 0.05 <= r[0] <= self.window[1] + 0.05]
            if not inside:  # region shorter than the sampling interval
                inside = [r for r in rows if r[0] <= self.window[1] + 0.05][-2:]
                where = "last samples before the end of the timed region"
        sm = [r[1] for r in inside]
        reasons = sorted({n for r in inside for n in r[3]})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": inside[-1][2] if inside else None,
                "reasons": reasons, "samples": len(sm), "window": where}


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), \
        int(os.environ.get("WORLD_SIZE", 1))


def max_over_ranks(value, device=None):
    """The largest of every rank's `value` (the identity without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world, units_per_step, steps, max_ms):
    """Units all ranks processed per second, timed by the slowest rank (weak
    scaling: every rank runs its own replica of the workload)."""
    return world * units_per_step * steps / (max_ms / 1e3)


def cpu_oracle_run(kind, B, H, T, D, sample_b, seed):
    """Time the fp64 oracle on host cores over `sample_b` batch rows of T tokens."""
    import torch
    if kind in ("glavl", "gdnvl"):  # a sample sequence of the pack
        kind = kind[:3]
    import oracle
    from paper_2606_01294_gb300 import inputs as gen
    if kind == "decode":
        Dd = gen.make_decode_inputs(gen.GLA, sample_b, H, D, D, seed=seed)
        pre = oracle.forward(gen.GLA, Dd["prefix"]["q"], Dd["prefix"]["k"], Dd["prefix"]["v"],
                             Dd["prefix"]["gate"], Dd["prefix"]["lam"])
        tk = Dd["token"]
        t0 = time.perf_counter()
        oracle.decode_step(gen.GLA, tk["q"], tk["k"], tk["v"], tk["gate"], tk["lam"],
                           pre["S"], pre["C"], pre["m"], pre["t"])
        dt = time.perf_counter() - t0
        return sample_b / dt, dt
    bb = gen.GDN if kind == "gdn" else gen.GLA
    P = gen.make_inputs(bb, sample_b, T, H, D, D, dtype=torch.bfloat16, seed=seed)
    G = gen.make_backward_inputs(sample_b, T, H, D, D, seed=seed + 1, state_grads=False) \
        if kind in ("glabwd", "gdnbwd") else None
    t0 = time.perf_counter()
    oracle.forward(bb, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"])
    if kind == "glabwd":
        oracle.gla_backward(P["q"], P["k"], P["v"], P["gate"], P["lam"], G["dout"])
    if kind == "gdnbwd":
        oracle.gdn_backward(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"], G["dout"])
    dt = time.perf_counter() - t0
    return sample_b * T / dt, dt


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return
    import oracle
    oracle.build_oracle()
    kind, B, H, T, D = WORKLOADS[args.workload]
    # one step = a bounded sample of the workload: one batch row (all heads)
    # over the first Ts tokens, so that warm-up + steps stay within minutes
    sample_b = 1 if kind != "decode" else 16
    Ts = min(T, 1024) if kind != "decode" else 1
    if kind in ("glavl", "gdnvl"):
        Ts = 1024
    cores = os.cpu_count() or 1
    for _ in range(args.warmup):
        cpu_oracle_run(kind, B, H, Ts, D, sample_b, seed=99)
    times = []
    for _ in range(args.steps):
        _, dt = cpu_oracle_run(kind, B, H, Ts, D, sample_b, seed=1236)
        times.append(dt)
    rate = sample_b * Ts * args.steps / sum(times)
    sample = (f"batch row 0 of {B}, all {H} heads, first {Ts} of {T} tokens, per step"
              if kind != "decode" else f"{sample_b} of {B} batch rows, all {H} heads, one token")
    line = {
        "impl": "reference", "metric": METRICS.get(kind, METRIC),
        "value": rate, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * statistics.mean(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.workload, "backbone": kind, "B": B, "H": H, "T": T,
                   "d_k": D, "d_v": D, "chunk": 64, "global_batch": B, "seq_len": T},
        "cpu_baseline": {"value": rate, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": rate, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def setup_workload(kind, B, H, T, D, dev, seed):
    """Inputs resident in HBM plus pinned host copies for one workload.  Returns
    (step, e2e_step, tokens_per_step, h2d_bytes, d2h_bytes): `step` runs one step on the
    device-resident inputs, `e2e_step` copies that step's inputs from pinned host memory,
    runs it and reads the result back."""
    import torch
    from paper_2606_01294_gb300 import ccq
    from paper_2606_01294_gb300 import inputs as gen

    if kind == "decode":
        Dd = gen.make_decode_inputs(gen.GLA, B, H, D, D, seed=seed)
        pre = {n: (None if x is None else x.to(dev)) for n, x in Dd["prefix"].items()}
        tok = {n: (None if x is None else x.to(dev)) for n, x in Dd["token"].items()}
        _, state0 = ccq.gla_fwd(pre["q"], pre["k"], pre["v"], pre["gate"], pre["lam"])
        state = ccq.CCQState(*(x.clone() for x in (state0.S, state0.C, state0.m, state0.t)))
        out = torch.empty(B, H, D, dtype=torch.bfloat16, device=dev)

        def step():
            ccq.decode_step(gen.GLA, tok["q"], tok["k"], tok["v"], tok["gate"], tok["lam"], state,
                            out=out)
        tokens_per_step = B
        host = {n: (None if x is None else x.pin_memory()) for n, x in Dd["token"].items()}
    elif kind == "glabwd":
        P = gen.make_inputs(gen.GLA, B, T, H, D, D, dtype=torch.bfloat16, seed=seed, lam="trained")
        P["dout"] = gen.make_backward_inputs(B, T, H, D, D, seed=seed + 1, state_grads=False)["dout"]
        Dv = {n: (None if x is None else x.to(dev)) for n, x in P.items()}
        out = torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev)
        fstate = ccq.CCQState.empty(B, H, D, D, dev)
        ws = ccq.gla_workspace(B, T, H, D, D, dev)
        ck = torch.empty(ccq.gla_ckpt_size(B, T, H, D, D), dtype=torch.uint8, device=dev)
        bws = ccq.gla_bwd_workspace(B, T, H, D, D, dev, with_ckpt=True)
        grads = {"dq": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dk": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dv": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dgk": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dlambda": torch.empty(B, T, H, device=dev),
                 "dS0": torch.empty(B, H, D, D, device=dev), "dC0": torch.empty(B, H, D, D, device=dev),
                 "dm0": torch.empty(B, H, D, device=dev)}

        def train_step(d):
            ccq.gla_fwd_save(d["q"], d["k"], d["v"], d["gate"], d["lam"], out=out, final_state=fstate,
                             workspace=ws, ckpt=ck)
            ccq.gla_bwd(d["q"], d["k"], d["v"], d["gate"], d["lam"], d["dout"], ckpt=ck, out=grads,
                        workspace=bws)

        def step():
            train_step(Dv)
        tokens_per_step = B * T
        host = {n: (None if x is None else x.pin_memory()) for n, x in P.items()}
    elif kind == "gdnbwd":
        P = gen.make_inputs(gen.GDN, B, T, H, D, D, dtype=torch.bfloat16, seed=seed, lam="trained")
        P["dout"] = gen.make_backward_inputs(B, T, H, D, D, seed=seed + 1, state_grads=False)["dout"]
        Dv = {n: (None if x is None else x.to(dev)) for n, x in P.items()}
        out = torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev)
        fstate = ccq.CCQState.empty(B, H, D, D, dev)
        ws = ccq.gdn_workspace(B, T, H, D, D, dev)
        bws = ccq.gdn_bwd_workspace(B, T, H, D, D, dev)
        grads = {"dq": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dk": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dv": torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev),
                 "dg": torch.empty(B, T, H, device=dev), "dbeta": torch.empty(B, T, H, device=dev),
                 "dlambda": torch.empty(B, T, H, device=dev),
                 "dS0": torch.empty(B, H, D, D, device=dev), "dC0": torch.empty(B, H, D, D, device=dev),
                 "dm0": torch.empty(B, H, D, device=dev)}

        def train_step(d):
            ccq.gdn_fwd(d["q"], d["k"], d["v"], d["gate"], d["beta"], d["lam"], out=out, final_state=fstate,
                        workspace=ws)
            ccq.gdn_bwd(d["q"], d["k"], d["v"], d["gate"], d["beta"], d["lam"], d["dout"], out=grads,
                        workspace=bws)

        def step():
            train_step(Dv)
        tokens_per_step = B * T
        host = {n: (None if x is None else x.pin_memory()) for n, x in P.items()}
    elif kind in ("glavl", "gdnvl"):
        bb = gen.GLA if kind == "glavl" else gen.GDN
        lens = varlen_lengths(B)
        total = sum(lens)
        cu = [0]
        for n in lens:
            cu.append(cu[-1] + n)
        P = {n: (None if x is None else x[0])
             for n, x in gen.make_inputs(bb, 1, total, H, D, D, dtype=torch.bfloat16, seed=seed).items()}
        Dv = {n: (None if x is None else x.to(dev)) for n, x in P.items()}
        out = torch.empty(total, H, D, dtype=torch.bfloat16, device=dev)
        fstate = ccq.CCQState.empty(B, H, D, D, dev)
        need = ccq.varlen_workspace_size(bb, cu, H, D, D)
        ws = torch.empty(max(need, 1), dtype=torch.uint8, device=dev)

        def run(d):
            o, _ = ccq.fwd_varlen(bb, d["q"], d["k"], d["v"], d["gate"], d["lam"], cu, beta=d["beta"], out=out,
                                  workspace=ws, final_state=fstate)
            return o

        def step():
            run(Dv)
        tokens_per_step = total
        host = {n: (None if x is None else x.pin_memory()) for n, x in P.items()}
    else:
        bb = gen.GLA if kind == "gla" else gen.GDN
        P = gen.make_inputs(bb, B, T, H, D, D, dtype=torch.bfloat16, seed=seed)
        Dv = {n: (None if x is None else x.to(dev)) for n, x in P.items()}
        out = torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev)
        fstate = ccq.CCQState.empty(B, H, D, D, dev)
        ws = (ccq.gdn_workspace if kind == "gdn" else ccq.gla_workspace)(B, T, H, D, D, dev)

        def step():
            if kind == "gla":
                ccq.gla_fwd(Dv["q"], Dv["k"], Dv["v"], Dv["gate"], Dv["lam"], out=out,
                            final_state=fstate, workspace=ws)
            else:
                ccq.gdn_fwd(Dv["q"], Dv["k"], Dv["v"], Dv["gate"], Dv["beta"], Dv["lam"], out=out,
                            final_state=fstate, workspace=ws)
        tokens_per_step = B * T
        host = {n: (None if x is None else x.pin_memory()) for n, x in P.items()}

    def e2e_step():
        d = {n: (None if x is None else x.to(dev, non_blocking=True)) for n, x in host.items()}
        if kind == "decode":
            o = ccq.decode_step(gen.GLA, d["q"], d["k"], d["v"], d["gate"], d["lam"], state, out=out)
            return o.to("cpu", non_blocking=True)
        if kind == "glabwd":
            train_step(d)
            return [grads[n].to("cpu", non_blocking=True) for n in ("dq", "dk", "dv", "dgk")]
        if kind == "gdnbwd":
            train_step(d)
            return [grads[n].to("cpu", non_blocking=True) for n in ("dq", "dk", "dv", "dg")]
        if kind in ("glavl", "gdnvl"):
            return run(d).to("cpu", non_blocking=True)
        if kind == "gla":
            o, _ = ccq.gla_fwd(d["q"], d["k"], d["v"], d["gate"], d["lam"], out=out,
                               final_state=fstate, workspace=ws)
        else:
            o, _ = ccq.gdn_fwd(d["q"], d["k"], d["v"], d["gate"], d["beta"], d["lam"], out=out,
                               final_state=fstate, workspace=ws)
        return o.to("cpu", non_blocking=True)

    h2d = sum(x.numel() * x.element_size() for x in host.values() if x is not None)
    d2h = out.numel() * out.element_size() * (4 if kind == "glabwd" else 1)
    if kind == "gdnbwd":
        d2h = sum(grads[n].numel() * grads[n].element_size() for n in ("dq", "dk", "dv", "dg"))
    return step, e2e_step, tokens_per_step, h2d, d2h


def time_steps(step, steps, warmup, dev, local_rank, world):
    """W untimed warm-up steps, then exactly K steps bracketed by a barrier and a
    synchronize, each step between two CUDA events on the launching stream; clocks sampled
    during the timed region.  Returns (total_ms max over ranks, per-step event ms, clocks)."""
    import torch
    import torch.distributed as dist
    from paper_2606_01294_gb300 import ccq
    stream = torch.cuda.current_stream(dev)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    with ClockSampler(local_rank) as clocks:
        time.sleep(0.3)  # nvidia-smi start-up
        for _ in range(warmup):
            step()
        ccq.device_status()
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        w0 = time.time()
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for i in range(steps):
            ev[i][0].record(stream)
            step()
            ev[i][1].record(stream)
        t_end.record(stream)
        torch.cuda.synchronize()
        clocks.window = (w0, time.time())
        time.sleep(0.1)
    if world > 1:
        dist.barrier()
    ccq.device_status()
    total_ms = max_over_ranks(t_start.elapsed_time(t_end), dev)
    return total_ms, [a.elapsed_time(b) for a, b in ev], clocks.summary()


def roofline(kind, workload, B, H, T, D, kern_ms, peaks):
    bytes_ = algorithmic_bytes(kind, B, H, T, D)
    achieved = bytes_ / (kern_ms / 1e3) / 1e9
    return {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / peaks["hbm_gbs"],
            "traffic": measured_traffic(kind, workload),
            "kernel": {"gla_bf16_20k": "whole step: gla_segment_state_kernel + gla_segment_combine_kernel"
                                       " + gla_chunk_kernel",
                       "gdn_bf16_20k": "whole step: gdn_wy_kernel + gdn_segment_state_kernel"
                                       " + gdn_segment_combine_kernel + gdn_chunk_kernel"}.get(
                           workload, KERNEL_NAMES[kind]), "algorithmic_bytes": bytes_,
            "peak_source": "measured (MEASURED_PEAKS.json hbm_gbs)",
            "flops": algorithmic_flops(kind, B, H, T, D)}


# Workloads the default run times beside the headline one (same steps and warm-up), each
# reported under "also" with its own roofline: the second T = 4096 forward configuration.
ALSO_DEFAULT = ("gdn_bf16_4k",)


def run_gpu(args):
    import torch
    import torch.distributed as dist

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    from __graft_entry__ import build
    if rank == 0 or world == 1:
        build()
    if world > 1:
        dist.barrier()
        build()

    kind, B, H, T, D = WORKLOADS[args.workload]
    if kind in ("glavl", "gdnvl"):
        T = sum(varlen_lengths(B))  # the packed length
    seed = 1236 + rank
    stream = torch.cuda.current_stream(dev)
    step, e2e_step, tokens_per_step, h2d, d2h = setup_workload(kind, B, H, T, D, dev, seed)
    total_ms, launch_ms, clock_summary = time_steps(step, args.steps, args.warmup, dev, local_rank, world)
    ms_per_step = total_ms / args.steps
    value = whole_job_rate(world, tokens_per_step, args.steps, total_ms)

    # ---------------- e2e: host buffers, copies inside the timed region
    e2e_steps = max(3, min(args.steps, 10))
    e2e_step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, dev)
    e2e_value = whole_job_rate(world, tokens_per_step, 1, e2e_ms)
    del step, e2e_step

    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    also = {}
    if args.workload == "gla_bf16_4k" and not args.no_also:
        for name in ALSO_DEFAULT:
            k2, B2, H2, T2, D2 = WORKLOADS[name]
            st2, _, tok2, _, _ = setup_workload(k2, B2, H2, T2, D2, dev, seed + 1)
            tot2, lms2, clk2 = time_steps(st2, args.steps, args.warmup, dev, local_rank, world)
            also[name] = {"ms_per_step": tot2 / args.steps,
                          "value": whole_job_rate(world, tok2, args.steps, tot2), "unit": "tokens/s",
                          "config": {"backbone": k2, "B": B2, "H": H2, "T": T2, "d_k": D2, "d_v": D2,
                                     "chunk": 64},
                          "gpu_launches": args.steps * launches_per_step(k2, B2, H2, T2, sms),
                          "kernel_ms_mean": statistics.mean(lms2), "clocks": clk2, "lms": lms2}
            del st2
            torch.cuda.empty_cache()

    line = None
    if rank == 0:
        with open(PEAKS_FILE) as f:
            peaks = json.load(f)
        kern_ms = statistics.mean(launch_ms)
        roof = roofline(kind, args.workload, B, H, T, D, kern_ms, peaks)
        for name, a in also.items():
            k2, B2, H2, T2, D2 = WORKLOADS[name]
            a["roofline"] = roofline(k2, name, B2, H2, T2, D2, a["kernel_ms_mean"], peaks)
            del a["lms"]
        cpu = None
        if not args.no_cpu_baseline and world == 1:
            import oracle
            oracle.build_oracle()
            # repeat passes over a bounded sample until about 10 s of CPU work
            sample_b = {"decode": 32, "glabwd": 1, "gdnbwd": 1, "glavl": 1, "gdnvl": 1}.get(kind, B)
            Tc = min(T, 1024) if kind in ("glabwd", "gdnbwd") else (1024 if kind in ("glavl", "gdnvl") else T)
            toks, secs, passes = 0.0, 0.0, 0
            while secs < 10.0 and passes < 20:
                rate, dt = cpu_oracle_run(kind, B, H, Tc, D, sample_b, seed=seed)
                toks += rate * dt
                secs += dt
                passes += 1
            cpu = {"value": toks / secs, "unit": "tokens/s", "cores": os.cpu_count(),
                   "kind": "oracle",
                   "sample": (f"{sample_b} of {B} batch rows, all {H} heads, {Tc} of {T} tokens, "
                              f"{passes} passes ({secs:.1f} s)")}
        line = {
            "metric": METRICS.get(kind, METRIC), "value": value,
            "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": args.workload, "backbone": kind, "B": B, "H": H, "T": T,
                       "d_k": D, "d_v": D, "chunk": 64, "global_batch": B * world, "seq_len": T,
                       "parallelism": f"replicas{world}",
                       "l2": "inputs larger than L2 (no flush)"},
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": args.steps * launches_per_step(kind, B, H, T, sms),
            "clocks": clock_summary,
            "kernel_ms_mean": kern_ms,
            "kernel_ms_min": min(launch_ms),
        }
        if kind in ("glavl", "gdnvl"):
            lens = varlen_lengths(B)
            line["config"]["seq_len"] = None
            line["config"]["packing"] = (f"{B} sequences of {min(lens)}-{max(lens)} tokens (seeded draw from "
                                         f"100-4000), packed [T, H, D], one launch")
        if also:
            line["also"] = also
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="gla_bf16_4k", choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-also", action="store_true",
                    help="time only the named workload (the default run also times gdn_bf16_4k)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
