"""Benchmark: the SAS attention layer on GB300 through the C ABI.

A step is one pass of the whole hot path over one batch of synthetic input:
the SAS attention forward (block summaries, query projection, selector scores,
log-gates, Top-K, gated block-sparse attention), followed by the dense GELU
MLP on the same tokens where the workload has one.  Default workload
(video-scale long-sequence attention): B=1, H=24, N=75600+512, d=128, b=64,
K=32, learned selector with d_sel=128 on block-correlated queries (R2),
attention only.  Inputs are seeded synthetic data resident in HBM; L2 is
flushed (256 MiB write) between timed steps, outside the timed events.

Prints one JSON line (rank 0).  --impl reference times the CPU oracle on a
bounded sample of the same workload instead.

Other workloads (--workload): tiny, dit and hires (SAS layer + MLP),
mlp_stress (the MLP sublayer alone), qwen3_4b_prefill / qwen3_4b_packed (GQA
prefill, given scores), and decode: the SAS decode step (Alg. 2 with
per-group block selection over a paged KV cache) of a Qwen3-4B-shaped layer
(32 query heads, 8 KV heads, d=128, b=64, K=32 = a 2048-token budget) at
--context tokens for --batch sequences, captured in a CUDA graph, next to
the dense decode of the same cache.
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

METRIC = "ms/layer and effective TFLOP/s on 1xGB300; % of bf16 tensor-core roofline"
UNIT = "TFLOP/s"

WORKLOADS = {
    # D = F = 0: no MLP in the step; attn False: the MLP alone
    "video": dict(B=1, H=24, N=75600 + 512, d=128, topk=32, d_sel=128, D=0, F=0,
                  name="video-scale long-sequence SAS attention: B=1 H=24 N=75600+512 (21x45x80 patches + 512 text "
                       "tokens; last block 16 tokens) d=128 b=64 K=32, learned selector d_sel=128, attention only"),
    "dit": dict(B=2, H=24, N=4096 + 512, d=128, topk=32, d_sel=128, D=3072, F=12288,
                name="DiT-scale causal SAS layer: B=2 H=24 N=4096+512 d=128 b=64 K=32, learned selector d_sel=128, "
                     "GELU MLP 9216x3072->12288->3072"),
    "tiny": dict(B=1, H=4, N=256, d=64, topk=32, d_sel=64, D=256, F=1024,
                 name="tiny SAS layer: B=1 H=4 N=256 d=64 K=32, MLP 256->1024->256"),
    "hires": dict(B=1, H=24, N=16384 + 512, d=128, topk=32, d_sel=128, D=3072, F=12288,
                  name="high-resolution causal SAS layer: B=1 H=24 N=16384+512 d=128 K=32, MLP 16896x3072->12288->3072"),
    "mlp_stress": dict(B=1, H=0, N=16384, d=128, topk=0, d_sel=128, D=3072, F=12288, attn=False,
                       name="MLP-sublayer stress: 16384 tokens x 3072 -> 12288 -> 3072 bf16, exact-erf GELU"),
    # GQA prefill (group-shared selection from given scores, one table per KV group)
    "qwen3_4b_prefill": dict(B=1, H=32, Hkv=8, N=32768, d=128, topk=32, d_sel=128, D=2560, F=9728,
                             name="Qwen3-4B-shaped GQA prefill layer: B=1 Hq=32 Hkv=8 N=32768 d=128 b=64 K=32 "
                                  "(2048-token budget), given R1 scores per KV group, GELU MLP "
                                  "32768x2560->9728->2560 (in place of the model's SwiGLU MLP)"),
    # the same layer on 32768 tokens packed from 12 sequences of geometric lengths
    "qwen3_4b_packed": dict(B=1, H=32, Hkv=8, N=32768, d=128, topk=32, d_sel=128, D=2560, F=9728,
                            lens=[16384, 8192, 4096, 2048, 1024, 512, 256, 128, 64, 32, 16, 16],
                            name="Qwen3-4B-shaped GQA prefill layer on 32768 packed tokens (12 sequences of "
                                 "16384, 8192, ..., 32, 16, 16 tokens): Hq=32 Hkv=8 d=128 b=64 K=32, given R1 "
                                 "scores per KV group, GELU MLP 32768x2560->9728->2560"),
}


def algorithmic_flops(w, learned=True):
    """Work the method itself must do for one layer (no tile-union or padding waste).

    Attention per (batch, head) row i with c = floor(i/64):
      4 d (|current-block keys| + 64 min(K, c))    QK^T and PV over the kept keys
      2 d_sel c                                    selector scores against c summaries
      2 d d_sel                                    query projection
    plus 2 d d_sel per full key block (key projection), and the MLP 4 T D F.
    With given scores (learned=False) the selector terms are not part of the layer.
    """
    N, d, K, ds = w["N"], w["d"], w["topk"], w["d_sel"]
    BH = w["B"] * w["H"]
    attn = sel = 0
    for c in range((N + 63) // 64):
        rows = min(64, N - 64 * c)
        cur = rows * (rows + 1) // 2            # sum over rows of (i - 64c + 1)
        attn += 4 * d * (cur + rows * 64 * min(K, c))
        sel += rows * (2 * ds * c + 2 * d * ds)
    sel += (N // 64) * 2 * d * ds
    if not learned:
        sel = 0
    if not w.get("attn", True):
        attn = sel = 0
    mlp = 4 * w["B"] * N * w["D"] * w["F"]
    return {"attention": BH * attn, "selector": BH * sel, "mlp": mlp,
            "total": BH * (attn + sel) + mlp}


def train_flops(w, form="sparse"):
    """(forward, backward) algorithmic FLOPs of one attention training step:
    the forward's 4 d per attended (row, key) pair and the backward's 10 d.
    form "full": the full training scope (every historical block kept: K = C_i
    in those counts); "ste": the hard Top-K gate under the straight-through
    estimator, whose gate pass adds q.k and dO.v (4 d) for every historical
    key of every row; "sparse": the SAS scope."""
    lens = w.get("lens")
    if lens:
        fl = packed_flops(w)
    else:
        C = (w["N"] + 63) // 64
        fl = algorithmic_flops(dict(w, topk=C) if form == "full" else w, learned=False)
    f_fwd = fl["attention"]
    f_bwd = f_fwd * 10 // 4
    if form == "ste":
        N, d = w["N"], w["d"]
        hist = sum(min(64, N - 64 * c) * 64 * c for c in range((N + 63) // 64))
        f_bwd += 4 * d * w["B"] * w["H"] * hist
    return f_fwd, f_bwd


def packed_flops(w, learned=False):
    """algorithmic_flops summed over the packed sequences (the MLP runs on all tokens)."""
    att = sel = 0
    for n in w["lens"]:
        if n > 0:
            f = algorithmic_flops(dict(w, N=n, B=1), learned)
            att += f["attention"]
            sel += f["selector"]
    mlp = 4 * w["N"] * w["D"] * w["F"]
    return {"attention": att, "selector": sel, "mlp": mlp, "total": att + sel + mlp}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"bf16": d.get("bf16_tflops"), "bf16_sustained": d.get("bf16_tflops_sustained"),
                "hbm": d.get("hbm_gbs"), "source": "measured"}
    return {"bf16": 1900.0, "bf16_sustained": 1700.0, "hbm": 6800.0, "source": "fallback"}


# ----------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ["clocks.sm", "clocks.max.sm", "utilization.gpu", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]

    def __init__(self, index):
        self.index = index
        self.rows = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) == len(self.FIELDS):
                self.rows.append(parts)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons = [], 0.0, set()
        for r in self.rows:
            try:
                clk, cmax, util = float(r[0]), float(r[1]), float(r[2])
            except ValueError:
                continue
            mx = max(mx, cmax)
            if util > 0:
                sm.append(clk)
            for k, name in enumerate(names):
                if r[3 + k].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx or None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------- multi-rank helpers

def reduce_max(values, dist, device):
    """Max of each value over all ranks (identity without a process group):
    the slowest rank sets the job's time."""
    if dist is None:
        return list(values)
    import torch
    t = torch.tensor(list(values), device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def job_throughput(tflop_per_step, world, ms_per_step):
    """Whole-job TFLOP/s: every rank runs one replica of the step (weak scaling)."""
    return tflop_per_step * world / (ms_per_step / 1e3)


# --------------------------------------------------------------- our arm

def kernel_traffic(kind, workload):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    this workload and the kernel's sources are unchanged since (else None)."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    rec = json.load(open(p)).get(kind)
    if not rec or rec.get("workload") != workload:
        return None
    m = hashlib.sha256()
    for f in rec["sources"]:
        m.update(open(os.path.join(ROOT, "paper_2609_13141_gb300", "csrc", f), "rb").read())
    return rec["dram_bytes_per_launch"] if m.hexdigest()[:16] == rec["sources_sha256_16"] else None


def run_ours(args, w, rank, world):
    import torch

    from paper_2609_13141_gb300 import sas, synth

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    B, H, N, d, K, ds, D, F = (w[k] for k in ("B", "H", "N", "d", "topk", "d_sel", "D", "F"))
    attn = w.get("attn", True)
    mlp = D > 0 and F > 0
    Hkv = w.get("Hkv", H)
    lens = w.get("lens")                          # packed sequences (B = 1, token axis of N rows)
    T = B * N
    learned = attn and args.regime == "R2" and Hkv == H and not lens   # GQA / packing take given scores
    Q = Kk = V = S = None
    if not attn:
        pass
    elif learned:
        # R2: block-correlated queries through the learned selector
        Q, Kk, V = synth.qkv(B, H, N, d, seed=rank, regime="R2")
    elif Hkv == H:
        # R1: block-coherent selector scores supplied by the caller
        Q, Kk, V = synth.qkv(B, H, N, d, seed=rank, regime="iid")
        S = synth.scores(B, H, N, (N + 63) // 64, seed=rank, regime="R1")
    else:
        Q = synth.qkv(B, H, N, d, seed=rank, regime="iid")[0]
        _, Kk, V = synth.qkv(B, Hkv, N, d, seed=rank + 100, regime="iid")
        S = synth.scores(B, Hkv, N, (max(lens) + 63) // 64 if lens else (N + 63) // 64, seed=rank, regime="R1")
    to = lambda t: None if t is None else t.to(dev)
    Qd, Kd, Vd, Sd = to(Q), to(Kk), to(V), to(S)
    Wqd = Wkd = None
    if learned:
        Wq, Wk = synth.selector_weights(H, d, ds, seed=rank)
        Wqd, Wkd = Wq.to(dev), Wk.to(dev)
    X = W1d = W2d = Xd = Yd = None
    if mlp:
        X, W1, W2, _, _ = synth.mlp(T, D, F, seed=rank)
        Xd, W1d, W2d = X.to(dev), W1.to(dev), W2.to(dev)
        Yd = torch.empty(T, D, device=dev, dtype=torch.bfloat16)
    Od = torch.empty_like(Qd) if attn else None
    LSEd = torch.empty(B, H, N, device=dev, dtype=torch.float32) if attn else None
    flush = torch.empty(256 * 1024 * 1024 // 4, device=dev, dtype=torch.float32)

    if not attn:
        layer = sas.SasLayer(1, 1, 64, 64, 0)     # a handle for the MLP entry point
    elif learned:
        layer = sas.SasLayer(B, H, N, d, K, selector=sas.SAS_SEL_MEANPOOL_PROJ, d_sel=ds)
    elif lens:
        layer = sas.SasLayer(1, H, N, d, K, selector=sas.SAS_SEL_SCORES_GIVEN, Hkv=Hkv, max_seqs=len(lens),
                             max_seqlen=max(lens))
    else:
        layer = sas.SasLayer(B, H, N, d, K, selector=sas.SAS_SEL_SCORES_GIVEN, Hkv=Hkv)
    h = layer.h
    stream = torch.cuda.current_stream(dev)
    cud = None
    if lens:
        import numpy as np
        cud = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dev)

    def step(Qx, Kx, Vx, Xx, O, Y, Sx=None):
        if attn and lens:
            sas.sas_attention_fwd_varlen(h, cud, Qx[0], Kx[0], Vx[0], Sx[0], O[0], LSEd[0], None, None, stream)
        elif attn and learned:
            sas.sas_attention_fwd(h, Qx, Kx, Vx, O, None, Wqd, Wkd, LSEd, None, None, stream)
        elif attn:
            sas.sas_attention_fwd(h, Qx, Kx, Vx, O, Sx, None, None, LSEd, None, None, stream)
        if mlp:
            sas.sas_mlp_fwd(h, Xx, W1d, W2d, Y, None, None, stream)

    for _ in range(max(args.warmup, 3)):
        step(Qd, Kd, Vd, Xd, Od, Yd, Sd)
    torch.cuda.synchronize()
    # keep the GPU busy for ~1 s so the clock sampler sees it under load
    t_end = time.time() + 1.0
    while time.time() < t_end:
        step(Qd, Kd, Vd, Xd, Od, Yd, Sd)
        torch.cuda.synchronize()

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.2)
    sas.sas_set_timing(h, True)
    launches0 = sas.sas_launch_count(h)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    for k in range(args.steps):
        flush.zero_()
        starts[k].record(stream)
        step(Qd, Kd, Vd, Xd, Od, Yd, Sd)
        ends[k].record(stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    launches = sas.sas_launch_count(h) - launches0
    kt = sas.sas_get_timings(h)
    # the attention kernel's executed work in the last forward: (128-row tile, 64-key block) products
    work_tiles, work_blocks = sas.sas_get_attention_work(h) if attn else (0, 0)
    sas.sas_set_timing(h, False)
    clocks = sampler.stop()
    ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / args.steps
    assert sas.sas_get_device_status(h) == 0, "device status word reports a timed-out wait"

    # end to end: pinned host inputs -> device -> layer -> host outputs, every step.
    # Heads are independent, so the step is streamed in head groups through the
    # same public calls: group g's inputs are copied in while group g - 1 is
    # computed and group g - 2's outputs are copied out (packed sequences and
    # the MLP-only workload run as one group).
    copies, outs = [], []
    dQ = dK = dV = dX = dS = None
    if attn:
        hQ, hK, hV = (t.pin_memory() for t in (Q, Kk, V))
        dQ, dK, dV = (torch.empty_like(t) for t in (Qd, Kd, Vd))
        hS = S.pin_memory() if S is not None else None
        if S is not None:
            dS = torch.empty_like(Sd)
        hO = torch.empty(Q.shape, dtype=torch.bfloat16).pin_memory()
    if mlp:
        dX = torch.empty_like(Xd)
        hX = X.pin_memory()
        hY = torch.empty(T, D, dtype=torch.bfloat16).pin_memory()
    G = H // Hkv if attn else 1
    max_groups = args.e2e_groups
    gk = Hkv if (not attn or lens) else next(k for k in range(1, Hkv + 1) if Hkv % k == 0 and B * Hkv // k <= max_groups)
    groups = [(b, kv0) for b in range(B) for kv0 in range(0, Hkv, gk)] if attn else []
    ghandle = None
    if attn and not lens:
        ghandle = sas.SasLayer(1, gk * G, N, d, K,
                               selector=sas.SAS_SEL_MEANPOOL_PROJ if learned else sas.SAS_SEL_SCORES_GIVEN,
                               d_sel=ds, Hkv=gk)
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in groups]
    ev_c = [torch.cuda.Event() for _ in groups]
    ev_x, ev_m = torch.cuda.Event(), torch.cuda.Event()
    LSEg = torch.empty(B, H, N, device=dev, dtype=torch.float32) if attn else None

    def e2e_step(k):
        flush.zero_()
        if k >= 0:
            e_st[k].record(stream)
        s_in.wait_stream(stream)
        with torch.cuda.stream(s_in):
            for gi, (b, kv0) in enumerate(groups):
                h0, h1, kv1 = kv0 * G, (kv0 + gk) * G, kv0 + gk
                dQ[b, h0:h1].copy_(hQ[b, h0:h1], non_blocking=True)
                dK[b, kv0:kv1].copy_(hK[b, kv0:kv1], non_blocking=True)
                dV[b, kv0:kv1].copy_(hV[b, kv0:kv1], non_blocking=True)
                if dS is not None:
                    dS[b, kv0:kv1].copy_(hS[b, kv0:kv1], non_blocking=True)
                ev_in[gi].record(s_in)
            if mlp:
                dX.copy_(hX, non_blocking=True)
                ev_x.record(s_in)
        for gi, (b, kv0) in enumerate(groups):
            h0, h1, kv1 = kv0 * G, (kv0 + gk) * G, kv0 + gk
            stream.wait_event(ev_in[gi])
            if lens:
                sas.sas_attention_fwd_varlen(h, cud, dQ[0], dK[0], dV[0], dS[0], Od[0], LSEd[0], None, None, stream)
            elif learned:
                sas.sas_attention_fwd(ghandle.h, dQ[b, h0:h1], dK[b, kv0:kv1], dV[b, kv0:kv1], Od[b, h0:h1], None,
                                      Wqd[h0:h1], Wkd[h0:h1], LSEg[b, h0:h1], None, None, stream)
            else:
                sas.sas_attention_fwd(ghandle.h, dQ[b, h0:h1], dK[b, kv0:kv1], dV[b, kv0:kv1], Od[b, h0:h1],
                                      dS[b, kv0:kv1], None, None, LSEg[b, h0:h1], None, None, stream)
            ev_c[gi].record(stream)
            s_out.wait_event(ev_c[gi])
            with torch.cuda.stream(s_out):
                hO[b, h0:h1].copy_(Od[b, h0:h1], non_blocking=True)
        if mlp:
            stream.wait_event(ev_x)
            sas.sas_mlp_fwd(h, dX, W1d, W2d, Yd, None, None, stream)
            ev_m.record(stream)
            s_out.wait_event(ev_m)
            with torch.cuda.stream(s_out):
                hY.copy_(Yd, non_blocking=True)
        stream.wait_stream(s_out)
        if k >= 0:
            e_en[k].record(stream)

    e_st = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e_en = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    for k in range(-2, args.steps):
        e2e_step(k)
    torch.cuda.synchronize()
    e2e_ms = sum(s.elapsed_time(e) for s, e in zip(e_st, e_en)) / args.steps
    h2d = sum(t.numel() * t.element_size() for t in (Q, Kk, V, S, X if mlp else None) if t is not None)
    d2h = (Q.numel() * 2 if attn else 0) + (T * D * 2 if mlp else 0)
    if ghandle is not None:
        assert sas.sas_get_device_status(ghandle.h) == 0
        ghandle.close()

    # tile-union statistics of the last forward (executed vs algorithmic work)
    unions = []
    if attn:
        Tt = (N + 127) // 128
        if lens:
            # packed: the first sum(ceil(n/128)) slots of each group are the tiles in use
            slots = (N + 127) // 128 + len(lens)
            used = sum((n + 127) // 128 for n in lens)
            allc = sas.sas_get_tile_union_counts(h, Hkv * slots)
            unions = [allc[g * slots + k] for g in range(Hkv) for k in range(used)]
        else:
            unions = sas.sas_get_tile_union_counts(h, B * Hkv * Tt)
    layer.close()

    ms, e2e_ms = reduce_max([ms, e2e_ms], dist, dev)
    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return None

    fl = packed_flops(w) if lens else algorithmic_flops(w, learned)
    tflop = fl["total"] / 1e12
    value = job_throughput(tflop, world, ms)
    # per kind: launches in the timed steps, time per launch and per step (a kind
    # may launch twice a step: head-packed tiles add the segment unions to the selection)
    per_kind = {k: {"launches": n, "ms_per_launch": (t / n if n else None), "ms_per_step": (t / args.steps if n else None)}
                for k, (n, t) in kt.items()}
    flops_per_launch = {"attention": fl["attention"], "mlp_up_gelu": fl["mlp"] / 2, "mlp_down": fl["mlp"] / 2}
    dom = max((k for k in kt if kt[k][0] > 0), key=lambda k: kt[k][1])
    peaks = load_peaks()
    roof = None
    if dom in flops_per_launch:
        avg = kt[dom][1] / kt[dom][0]
        achieved = flops_per_launch[dom] / (avg / 1e3) / 1e12
        roof = {"bound": "tensor", "kernel": dom, "achieved": round(achieved, 1), "peak": peaks["bf16"],
                "unit": "TFLOP/s", "frac": round(achieved / peaks["bf16"], 4), "traffic": kernel_traffic(dom, w["name"]),
                "peak_source": f"{peaks['source']} bf16 dense burst"}
    out = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": ("synthetic (seeded; N(0,1) X, weights N(0,0.02))" if not attn else
                 "synthetic (seeded; R2 block-correlated queries q_i = (mu[block] + 0.3 eps_i)/sqrt(1.09), "
                 "N(0,1) K/V" + ("/X" if mlp else "") + ", weights N(0,0.02))" if learned else
                 "synthetic (seeded; R1 block-coherent selector scores s = u[block] + 0.05 eps given by the caller, "
                 "N(0,1) Q/K/V" + ("/X" if mlp else "") + ", weights N(0,0.02))"),
        "config": {"workload": w["name"], "B": B, "H": H, "Hkv": Hkv, "N": N, "d": d, "block": 64, "topk": K,
                   "d_sel": ds, "packed_lengths": lens,
                   "mlp": [T, D, F, D] if mlp else None,
                   "selector": None if not attn else ("meanpool_proj (R2)" if learned else "scores_given (R1)"),
                   "l2": "flushed between timed steps (256 MiB write)",
                   "parallelism": f"replicas x{world}"},
        "roofline": roof,
        "kernels": per_kind,
        "algorithmic_tflop_per_step": round(tflop, 4),
        "e2e": {"value": round(job_throughput(tflop, world, e2e_ms), 2), "unit": UNIT, "ms_per_step": round(e2e_ms, 4),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "streamed_head_groups": len(groups) if attn else 1},
        "gpu_launches": launches,
        "clocks": clocks,
    }
    if attn:
        # the SAS attention kernel proper: algorithmic work (each row's kept keys)
        # and executed work (every 128-row tile over the blocks it visits)
        a_avg = kt["attention"][1] / max(kt["attention"][0], 1)
        exe = work_blocks * 4 * 128 * 64 * d
        a_alg = fl["attention"] / (a_avg / 1e3) / 1e12
        a_exe = exe / (a_avg / 1e3) / 1e12
        sas_ms = sum(kt[k][1] / args.steps for k in ("block_summaries", "selection", "attention"))
        out["attention_kernel"] = {
            "ms": round(a_avg, 4), "algorithmic_tflops": round(a_alg, 1),
            "frac_of_bf16_peak": round(a_alg / peaks["bf16"], 4),
            "executed_tflop": round(exe / 1e12, 4), "executed_tflops": round(a_exe, 1),
            "executed_frac_of_bf16_peak": round(a_exe / peaks["bf16"], 4),
            "tiles": work_tiles,
            "mean_visited_blocks_per_tile": round(work_blocks / max(work_tiles, 1), 2),
            "mean_union_blocks_per_tile": round(sum(unions) / max(len(unions), 1), 2)}
        out["sas_layer"] = {"ms": round(sas_ms, 4),
                            "algorithmic_tflops": round((fl["attention"] + fl["selector"]) / (sas_ms / 1e3) / 1e12, 1),
                            "selection_ms": round(kt["selection"][1] / args.steps, 4),
                            "block_summaries_ms": round(kt["block_summaries"][1] / args.steps, 4)}
    if not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(w, budget_s=args.cpu_budget, learned=learned, workload=args.workload,
                                           topk=args.topk)
    if dist is not None:
        dist.destroy_process_group()
    return out


# ----------------------------------------------------------- CPU oracle

def _nproc():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def _oracle_threads():
    """Threads the oracle's matrix products may use (its BLAS pool; the
    per-row loops are single-threaded Python)."""
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 1) for i in threadpool_info()]
        return max(n) if n else 1
    except Exception:
        for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
            if os.environ.get(var, "").isdigit():
                return int(os.environ[var])
        return _nproc()


def oracle_sample(w, budget_s, seed=0, learned=True):
    """Runs the oracle on a bounded sample of the workload and returns its
    throughput on the workload's FLOP mix.

    The attention part runs query rows of one head (selector scores for the
    whole head, or the head's given R1 scores, then the gated attention of
    random rows); the MLP part runs random token rows.  With both, each gets
    half the budget and its rate (algorithmic FLOPs per second) is measured on
    its own; the full step's time is extrapolated as attention FLOPs /
    attention rate + MLP FLOPs / MLP rate.  Returns (rate_flops_per_s,
    seconds, desc)."""
    import numpy as np
    import torch

    from oracle import sas_oracle as OR
    from paper_2609_13141_gb300 import synth

    B, H, N, d, K, ds, D, F = (w[k] for k in ("B", "H", "N", "d", "topk", "d_sel", "D", "F"))
    attn, mlp = w.get("attn", True), D > 0 and F > 0
    share = budget_s / 2 if (attn and mlp) else budget_s
    f = lambda t: t.to(torch.float64).numpy()
    rng = np.random.default_rng(seed)
    parts = []
    a_time = m_time = 0.0
    a_rate = m_rate = None
    if attn:
        Q, Kk, V = synth.qkv(1, 1, N, d, seed=seed, regime="R2")
        Wq, Wk = synth.selector_weights(1, d, ds, seed=seed)
        q, k, v, wq, wk = f(Q[0, 0]), f(Kk[0, 0]), f(V[0, 0]), f(Wq[0]), f(Wk[0])
        if learned:
            t0 = time.perf_counter()
            s = OR.selector_scores(q, k, wq, wk, 64)
            a_flops = N * 2 * d * ds + (N // 64) * 2 * d * ds
        else:
            s = f(synth.scores(1, 1, N, (N + 63) // 64, seed=seed, regime="R1")[0, 0])
            t0 = time.perf_counter()
            a_flops = 0
        rows_done = 0
        while time.perf_counter() - t0 < share:
            rows = rng.integers(0, N, size=32)
            OR.sas_attention_head(q, k, v, s, 64, K, rows=rows)
            a_flops += sum(OR.attention_flops_row(int(i), 64, K, d, ds if learned else 0) for i in rows)
            rows_done += len(rows)
        a_time = time.perf_counter() - t0
        # the whole head's selector is amortised over the rows actually run
        a_rate = a_flops / a_time
        how = "with that head's selector" if learned else "with that head's given R1 scores"
        parts.append(f"{rows_done} random query rows of one head ({how}) in {a_time:.1f} s")
    if mlp:
        X, W1, W2, _, _ = synth.mlp(256, D, F, seed=seed)
        x, w1, w2 = f(X), f(W1), f(W2)
        t1 = time.perf_counter()
        m_flops = 0
        tok_done = 0
        while time.perf_counter() - t1 < share:
            toks = rng.integers(0, 256, size=2)
            OR.gelu_mlp(x, w1, w2, rows=toks)
            m_flops += 4 * len(toks) * D * F
            tok_done += len(toks)
        m_time = time.perf_counter() - t1
        m_rate = m_flops / m_time
        parts.append(f"{tok_done} MLP token rows in {m_time:.1f} s")

    fl = packed_flops(w) if w.get("lens") else algorithmic_flops(w, learned)
    full_time = ((fl["attention"] + fl["selector"]) / a_rate if attn else 0.0) + (fl["mlp"] / m_rate if mlp else 0.0)
    rate = fl["total"] / full_time
    desc = "oracle (numpy fp64): " + " and ".join(parts)
    if attn and mlp:
        desc += "; the two measured rates are combined by the layer's FLOP mix"
    desc += "; the full step's time is extrapolated from the sampled rate"
    return rate, a_time + m_time, desc


def _oracle_sample_one_thread(workload, budget_s, learned, topk):
    """oracle_sample in a fresh process whose BLAS pools are pinned to one
    thread (the variables are read when numpy loads, so it needs its own
    process).  Returns the rate in FLOP/s, or None if the run fails."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, os.path.abspath(__file__), "--oracle-sample-only", "--workload", workload,
           "--cpu-budget", str(budget_s), "--regime", "R2" if learned else "R1"]
    if topk is not None:
        cmd += ["--topk", str(topk)]
    try:
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=budget_s * 4 + 120)
        return json.loads(r.stdout.strip().splitlines()[-1])["rate"]
    except Exception:
        return None


def cpu_baseline(w, budget_s=12.0, learned=True, workload=None, topk=None):
    """The oracle timed on this host: once with its BLAS pool on every core
    (`value`), once pinned to one thread (`value_1_thread`), half the budget
    each."""
    rate, dt, desc = oracle_sample(w, budget_s / 2, learned=learned)
    one = _oracle_sample_one_thread(workload, budget_s / 2, learned, topk) if workload else None
    return {"value": round(rate / 1e12, 8), "unit": UNIT, "cores": _nproc(),
            "threads": _oracle_threads(), "kind": "oracle",
            "value_1_thread": None if one is None else round(one / 1e12, 8),
            "sample": desc + f"; matrix products on a BLAS pool of {_oracle_threads()} threads, per-row loops "
                             "single-threaded; value_1_thread: the same sample with the pool pinned to one thread",
            "seconds": round(dt, 2)}


def run_reference(args, w, rank, world):
    if rank != 0:
        return None
    rates = []
    desc = ""
    learned = args.regime == "R2" and w.get("Hkv", w["H"]) == w["H"] and not w.get("lens")   # as our arm
    for k in range(args.warmup + args.steps):
        rate, dt, desc = oracle_sample(w, budget_s=args.ref_step_s, seed=k, learned=learned)
        if k >= args.warmup:
            rates.append(rate)
    # harmonic mean: total FLOPs over total time for equal-work steps
    value = len(rates) / sum(1.0 / r for r in rates) / 1e12
    full = (packed_flops(w) if w.get("lens") else algorithmic_flops(w, learned))["total"]
    ms = full / (value * 1e12) * 1e3
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 8), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 2),
        "ms_per_step_extrapolated": True, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)",
        "config": {"workload": w["name"], "B": w["B"], "H": w["H"], "N": w["N"], "d": w["d"], "topk": w["topk"]},
        "cpu_baseline": {"value": round(value, 8), "unit": UNIT, "cores": _nproc(), "threads": _oracle_threads(),
                         "kind": "oracle",
                         "sample": desc + f"; each step a {args.ref_step_s:.0f}-second sample; ms_per_step is the "
                                          "whole step's FLOPs at the sampled rate (extrapolated, not run in full)"},
        "e2e": {"value": round(value, 8), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


# ------------------------------------------------------------ training step

TRAIN_METRIC = "SAS attention training step (forward + backward) of one layer: ms and TFLOP/s on 1xGB300"


def run_train(args, w, rank, world):
    """Forward + backward of the SAS attention (Alg. 1 steps 1-4 and Alg. 4) on
    the workload's attention shape, given block-coherent scores (R1) so that
    the score gradient is produced too; GQA workloads share K, V, the kept
    sets and the gates per KV group, packed ones run every sequence as its own
    problem.  Algorithmic FLOPs: the forward's 4 d per attended (row, key)
    pair plus the backward's 10 d (QK^T, dO V^T, dS K, dS^T Q, P^T dO).
    --train-form full: the full training scope (every historical block kept
    and gated: K = C_i in those counts).  --train-form ste: the hard Top-K gate
    under the straight-through estimator (the hard forward and backward, plus
    the gate gradient of every historical key: q.k and dO.v, 4 d a pair)."""
    import numpy as np
    import torch

    from paper_2609_13141_gb300 import sas, synth

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    B, H, N, d, K = (w[k] for k in ("B", "H", "N", "d", "topk"))
    Hkv = w.get("Hkv", H)
    lens = w.get("lens")
    C = ((max(lens) if lens else N) + 63) // 64
    Q = synth.qkv(B, H, N, d, seed=rank)[0]
    _, Kk, V = synth.qkv(B, Hkv, N, d, seed=rank + 100)
    S = synth.scores(B, Hkv, N, C, seed=rank, regime="R1")
    dO = synth.normal((B, H, N, d), rank + 5).to(torch.bfloat16)
    Qd, Kd, Vd, Sd, dOd = (t.to(dev) for t in (Q, Kk, V, S, dO))
    form = args.train_form
    if form != "sparse" and lens:
        raise SystemExit("--train-form full / ste take [B, H, N, d] workloads")
    if lens:
        layer = sas.SasLayer(1, H, N, d, K, selector=sas.SAS_SEL_SCORES_GIVEN, Hkv=Hkv, max_seqs=len(lens),
                             max_seqlen=max(lens))
        cud = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dev)
    else:
        layer = sas.SasLayer(B, H, N, d, K, selector=sas.SAS_SEL_SCORES_GIVEN, Hkv=Hkv,
                             mode=sas.SAS_MODE_TRAIN_HARD_STE if form == "ste" else sas.SAS_MODE_TRAIN_SOFT,
                             scope=sas.SAS_SCOPE_FULL if form == "full" else sas.SAS_SCOPE_SPARSE)
    h = layer.h
    stream = torch.cuda.current_stream(dev)
    O = torch.empty_like(Qd)
    LSE = torch.empty(B, H, N, device=dev, dtype=torch.float32)
    si = torch.empty(B, Hkv, N, max(K, 1), device=dev, dtype=torch.int32)
    sl = torch.empty(B, Hkv, N, max(K, 1), device=dev, dtype=torch.float32)
    dQ, dK, dV = torch.empty_like(Qd), torch.empty_like(Kd), torch.empty_like(Vd)
    dl = torch.empty_like(sl) if form == "sparse" else torch.empty(B, Hkv, N, C, device=dev, dtype=torch.float32)
    ds = torch.empty_like(Sd)
    if form == "full":
        si = sl = None   # the full scope keeps no Top-K
    flush = torch.empty(256 * 1024 * 1024 // 4, device=dev, dtype=torch.float32)

    def step():
        if lens:
            sas.sas_attention_fwd_varlen(h, cud, Qd[0], Kd[0], Vd[0], Sd[0], O[0], LSE[0], si[0], sl[0], stream)
        else:
            sas.sas_attention_fwd(h, Qd, Kd, Vd, O, Sd, None, None, LSE, si, sl, stream)
        sas.sas_attention_bwd(h, Qd, Kd, Vd, O, LSE, dOd, dQ, dK, dV, Sd, si, sl, dl, ds, stream)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.2)
    sas.sas_set_timing(h, True)
    l0 = sas.sas_launch_count(h)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for k in range(args.steps):
        flush.zero_()
        ev[k][0].record(stream)
        step()
        ev[k][1].record(stream)
    torch.cuda.synchronize()
    launches = sas.sas_launch_count(h) - l0
    kt = sas.sas_get_timings(h)
    sas.sas_set_timing(h, False)
    clocks = sampler.stop()
    assert sas.sas_get_device_status(h) == 0
    ms = sum(a.elapsed_time(b) for a, b in ev) / args.steps
    Tt = (N + 127) // 128 + (len(lens) if lens else 0)
    unions = sas.sas_get_tile_union_counts(h, B * Hkv * Tt)
    if lens:
        # packed: the first sum(ceil(n/128)) slots of each group are the tiles in use
        used = sum((n + 127) // 128 for n in lens)
        unions = [unions[g * Tt + k] for g in range(Hkv) for k in range(used)]
    layer.close()
    f_fwd, f_bwd = train_flops(w, form)
    tflop = (f_fwd + f_bwd) / 1e12
    peaks = load_peaks()
    # per step (the hard-STE backward is two launches of its kind, head-packed
    # selection two: the Top-K and the segment unions)
    bwd_ms = kt["attention_bwd"][1] / args.steps
    fwd_ms = kt["attention"][1] / args.steps
    sel_ms = kt["selection"][1] / args.steps
    ach = f_bwd / (bwd_ms / 1e3) / 1e12
    return {
        "metric": TRAIN_METRIC, "value": round(tflop / (ms / 1e3), 2), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16 (fp32 softmax and gradients of log g, s)",
        "data": "synthetic (seeded; R1 block-coherent scores given, N(0,1) Q/K/V/dO)",
        "config": {"workload": w["name"] + " (attention only, forward + backward)"
                   + {"sparse": "", "full": ", full training scope", "ste": ", hard Top-K gate with STE"}[form],
                   "B": B, "H": H, "Hkv": Hkv, "N": N, "d": d, "topk": K, "packed_lengths": lens, "form": form,
                   "l2": "flushed between timed steps (256 MiB write)", "parallelism": f"replicas x{world}"},
        "roofline": {"bound": "tensor", "kernel": "attention_bwd", "achieved": round(ach, 1), "peak": peaks["bf16"],
                     "unit": "TFLOP/s", "frac": round(ach / peaks["bf16"], 4), "traffic": None,
                     "peak_source": f"{peaks['source']} bf16 dense burst"},
        "mean_union_blocks_per_tile": round(sum(unions) / max(len(unions), 1), 2),
        "kernels_ms": {"selection": round(sel_ms, 4), "attention_fwd": round(fwd_ms, 4), "attention_bwd": round(bwd_ms, 4)},
        "algorithmic_tflop_per_step": round(tflop, 4),
        "gpu_launches": launches,
        "clocks": clocks,
    }


# ---------------------------------------------------------------- decode

DECODE_METRIC = "decode step latency of one attention layer (us), SAS vs dense, 1xGB300"


def decode_bytes(B, Hq, Hkv, d, ds, K, n, dense):
    """Algorithmic HBM bytes of one decode step and of each kernel kind for B
    sequences of n cached tokens (new token included)."""
    G = Hq // Hkv
    C = (n - 1) // 64
    cur = n - 64 * C
    groups = B * Hkv
    kv_tokens = (C if dense else min(K, C)) * 64 + cur
    attn = groups * (2 * 2 * kv_tokens * d + 2 * G * d * 2)           # K, V pages; q in, O out
    prep = groups * 4 * 2 * d                                         # k_new, v_new read and written
    if dense:
        return {"prep": prep, "attention": attn, "total": prep + attn}
    prep += groups * (2 * ds * G * d + 2 * G * d)                    # Wq and q for the gate query
    select = groups * (2 * C * ds + 2 * ds)                          # the summaries and q~
    return {"prep": prep, "select": select, "attention": attn, "total": prep + select + attn}


def decode_oracle_us(B, Hq, Hkv, d, ds, K, n, budget_s, seed=0):
    """Oracle (numpy fp64) time of one decode step, from groups run on the host
    cores until the budget is spent, scaled to the B*Hkv groups of a step."""
    import numpy as np
    import torch

    from oracle import decode_oracle as DO
    from paper_2609_13141_gb300 import synth

    G = Hq // Hkv
    nb = -(-n // 64)
    Kc, Vc = synth.decode_cache(nb, 1, d, seed=seed)
    q, _, _ = synth.decode_queries(1, G, 1, d, seed=seed)
    Wq, Wk = synth.decode_selector_weights(1, G, d, ds, seed=seed)
    f = lambda t: t.to(torch.float64).numpy()
    Kx = f(Kc[:, 0].reshape(-1, d))[:n]
    Vx = f(Vc[:, 0].reshape(-1, d))[:n]
    qx, wq, wk = f(q[0]), f(Wq[0]), f(Wk[0])
    t0 = time.perf_counter()
    done = 0
    while time.perf_counter() - t0 < budget_s or done == 0:
        DO.decode_group(qx, Kx, Vx, wq, wk, 64, K)
        done += 1
    per_group = (time.perf_counter() - t0) / done
    desc = (f"oracle (numpy fp64): {done} decode steps of one KV group ({G} query heads, {n} cached tokens, "
            f"selector + Top-K + attention) in {per_group * done:.1f} s, scaled to the {B * Hkv} groups of a step")
    return per_group * B * Hkv * 1e6, per_group * done, desc


def run_decode(args, rank, world):
    import torch

    from paper_2609_13141_gb300 import sas, synth

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    B, Hq, Hkv, d, ds = args.batch, 32, 8, 128, 128
    K = args.topk if args.topk is not None else 32
    n = args.context
    G = Hq // Hkv
    max_blocks = -(-n // 64)
    table, P = synth.decode_layout([n] * B, max_blocks, seed=rank)
    Kc, Vc = synth.decode_cache(P, Hkv, d, seed=rank, device=dev)
    q, kn, vn = synth.decode_queries(B, Hq, Hkv, d, seed=rank, device=dev)
    Wq, Wk = synth.decode_selector_weights(Hkv, G, d, ds, seed=rank, device=dev)
    Ksum = torch.zeros(B, Hkv, max_blocks, ds, device=dev, dtype=torch.bfloat16)
    tab = table.to(dev)
    lens = torch.full((B,), n, dtype=torch.int32, device=dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, device=dev, dtype=torch.float32)
    stream = torch.cuda.Stream(dev)

    def measure(dense):
        dec = sas.SasDecoder(B, Hq, Hkv, d, K, max_blocks, P, d_sel=ds, dense=dense)
        if not dense:
            dec.summarize(Kc, tab, lens - 1, Wk, Ksum)
        out = (torch.empty(B, Hq, d, device=dev, dtype=torch.bfloat16),
               torch.empty(B, Hq, device=dev, dtype=torch.float32),
               None if dense else torch.empty(B, Hkv, max(K, 1), device=dev, dtype=torch.int32))
        args_ = (q, Kc, Vc, tab, lens, kn, vn, Wq, Wk, None if dense else Ksum)
        with torch.cuda.stream(stream):
            for _ in range(max(args.warmup, 3)):
                dec.step(*args_, out=out, stream=stream)
            # one timed step outside capture creates the timing events, so the
            # capture below records existing events only
            sas.sas_decode_set_timing(dec.h, True)
            dec.step(*args_, out=out, stream=stream)
        stream.synchronize()
        # graph_t carries event nodes between the kernels for the per-kernel
        # breakdown; they serialise the kernels, so the step itself is timed on
        # a second graph without them (the kernels then overlap their set-up)
        sas.sas_decode_set_timing(dec.h, True)
        graph_t = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph_t, stream=stream):
            dec.step(*args_, out=out, stream=stream)
        sas.sas_decode_set_timing(dec.h, False)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            dec.step(*args_, out=out, stream=stream)
        launches_per_step = 2 if dense else 3
        for _ in range(max(args.warmup, 3)):
            graph.replay()
            graph_t.replay()
        torch.cuda.synchronize()
        per_kind = {}
        with torch.cuda.stream(stream):
            for k in range(args.steps):
                flush.zero_()
                graph_t.replay()
                stream.synchronize()
                for kind, (cnt, ms) in sas.sas_decode_get_timings(dec.h).items():
                    if cnt:
                        per_kind.setdefault(kind, []).append(ms)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        with torch.cuda.stream(stream):
            for k in range(args.steps):
                flush.zero_()
                ev[k][0].record(stream)
                graph.replay()
                ev[k][1].record(stream)
        torch.cuda.synchronize()
        per_step = sorted(a.elapsed_time(b) * 1e3 for a, b in ev)
        us = sum(per_step) / args.steps
        spread = {"min": round(per_step[0], 2), "median": round(per_step[len(per_step) // 2], 2),
                  "max": round(per_step[-1], 2)}
        assert sas.sas_decode_get_device_status(dec.h) == 0
        # end to end: the step's inputs from pinned host memory, its output back
        hq, hkn, hvn = q.cpu().pin_memory(), kn.cpu().pin_memory(), vn.cpu().pin_memory()
        hO = torch.empty(B, Hq, d, dtype=torch.bfloat16).pin_memory()
        e2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        with torch.cuda.stream(stream):
            for k in range(-2, args.steps):
                flush.zero_()
                if k >= 0:
                    e2[k][0].record(stream)
                q.copy_(hq, non_blocking=True)
                kn.copy_(hkn, non_blocking=True)
                vn.copy_(hvn, non_blocking=True)
                graph.replay()
                hO.copy_(out[0], non_blocking=True)
                if k >= 0:
                    e2[k][1].record(stream)
        torch.cuda.synchronize()
        e2e_us = sum(a.elapsed_time(b) for a, b in e2) / args.steps * 1e3
        dec.close()
        kern = {k: sum(v) / len(v) * 1e3 for k, v in per_kind.items()}
        h2d = (q.numel() + kn.numel() + vn.numel()) * 2
        return us, e2e_us, kern, launches_per_step * args.steps, h2d, hO.numel() * 2, spread

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.2)
    if args.decode_only == "dense":
        us, e2e_us, kern, launches, h2d, d2h, spread = measure(True)
    else:
        us, e2e_us, kern, launches, h2d, d2h, spread = measure(False)
    if args.decode_only is None:
        dus, de2e_us, dkern, _, _, _, dspread = measure(True)
    else:   # one arm only (profiling runs): the other arm's fields repeat it
        dus, de2e_us, dkern, dspread = us, e2e_us, kern, spread
    clocks = sampler.stop()
    us, e2e_us, dus = reduce_max([us, e2e_us, dus], dist, dev)
    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return None
    peaks = load_peaks()
    by = decode_bytes(B, Hq, Hkv, d, ds, K, n, args.decode_only == "dense")
    dby = decode_bytes(B, Hq, Hkv, d, ds, K, n, True) if args.decode_only is None else by

    def roof(kern_us, bytes_):
        dom = max(kern_us, key=kern_us.get)
        ach = bytes_[dom] / (kern_us[dom] / 1e6) / 1e9
        return {"bound": "hbm", "kernel": dom, "achieved": round(ach, 1), "peak": peaks["hbm"], "unit": "GB/s",
                "frac": round(ach / peaks["hbm"], 4), "traffic": None,
                "peak_source": f"{peaks['source']} HBM copy bandwidth"}

    wname = (f"Qwen3-4B-shaped decode attention layer: Hq=32 Hkv=8 d=128 b=64, K={K} ({K * 64}-token budget), "
             f"context {n} tokens, batch {B}, paged KV cache (one 64-token block per page)")
    out = {
        "metric": DECODE_METRIC, "value": round(us, 2), "unit": "us", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(us / 1e3, 5), "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 (fp32 scores/softmax)",
        "data": "synthetic (seeded; block-coherent keys, N(0,1) queries/values, selector weights N(0,0.02))",
        "config": {"workload": wname, "B": B, "Hq": Hq, "Hkv": Hkv, "d": d, "d_sel": ds, "topk": K, "context": n,
                   "graph": "one CUDA graph per step", "l2": "flushed between timed steps (256 MiB write)",
                   "parallelism": f"replicas x{world}"},
        "roofline": roof(kern, by),
        "kernels_us": {k: round(v, 2) for k, v in kern.items()},
        "step_us_spread": spread,
        "step_algorithmic_bytes": by["total"],
        "step_gbs": round(by["total"] / (us / 1e6) / 1e9, 1),
        "dense": {"us": round(dus, 2), "e2e_us": round(de2e_us, 2), "step_us_spread": dspread, "kernels_us": {k: round(v, 2) for k, v in dkern.items()},
                  "roofline": roof(dkern, dby), "step_algorithmic_bytes": dby["total"],
                  "step_gbs": round(dby["total"] / (dus / 1e6) / 1e9, 1)},
        "speedup_vs_dense": round(dus / us, 2),
        "e2e": {"value": round(e2e_us, 2), "unit": "us", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "clocks": clocks,
    }
    if not args.no_cpu_baseline:
        v, secs, desc = decode_oracle_us(B, Hq, Hkv, d, ds, K, n, args.cpu_budget / 2)
        out["cpu_baseline"] = {"value": round(v, 1), "unit": "us", "cores": _nproc(), "threads": _oracle_threads(), "kind": "oracle",
                               "sample": desc, "seconds": round(secs, 2)}
    if dist is not None:
        dist.destroy_process_group()
    return out


def run_decode_reference(args, rank, world):
    if rank != 0:
        return None
    K = args.topk if args.topk is not None else 32
    vals = []
    desc = ""
    for k in range(args.warmup + args.steps):
        v, _, desc = decode_oracle_us(args.batch, 32, 8, 128, 128, K, args.context, args.ref_step_s / 4, seed=k)
        if k >= args.warmup:
            vals.append(v)
    value = sum(vals) / len(vals)
    return {
        "impl": "reference", "metric": DECODE_METRIC, "value": round(value, 1), "unit": "us", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(value / 1e3, 3), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)",
        "config": {"workload": f"Qwen3-4B-shaped decode attention layer, context {args.context}, batch {args.batch}",
                   "B": args.batch, "context": args.context, "topk": K},
        "cpu_baseline": {"value": round(value, 1), "unit": "us", "cores": _nproc(), "threads": _oracle_threads(), "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": round(value, 1), "unit": "us", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS) + ["decode"], default="video")
    ap.add_argument("--context", type=int, default=65536, help="decode: cached tokens per sequence")
    ap.add_argument("--batch", type=int, default=1, help="decode: sequences per step")
    ap.add_argument("--decode-only", choices=["sparse", "dense"], default=None,
                    help="decode: run one arm only (for profiling)")
    ap.add_argument("--train", action="store_true",
                    help="time the attention training step (forward + backward) of the workload instead")
    ap.add_argument("--train-form", choices=["sparse", "full", "ste"], default="sparse",
                    help="--train: the sparse scope (SAS), the full training scope, or the hard Top-K gate with STE")
    ap.add_argument("--regime", choices=["R2", "R1"], default="R2",
                    help="R2: learned selector on block-correlated queries; R1: block-coherent scores given")
    ap.add_argument("--topk", type=int, default=None, help="override the workload's K")
    ap.add_argument("--heads", type=int, default=None,
                    help="override the workload's head count (smaller cases of the same shape, for profiling)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--ref-step-s", type=float, default=4.0)
    ap.add_argument("--oracle-sample-only", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--e2e-groups", type=int, default=8, help=argparse.SUPPRESS)   # streamed head groups, at most
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if args.workload == "decode":
        out = run_decode_reference(args, rank, world) if args.impl == "reference" else run_decode(args, rank, world)
        if out is not None and rank == 0:
            print(json.dumps(out))
        return
    w = dict(WORKLOADS[args.workload])
    if args.topk is not None:
        w["topk"] = args.topk
        w["name"] = w["name"].replace("K=32", f"K={args.topk}")
    if args.heads is not None:
        if w.get("Hkv", w["H"]) != w["H"]:
            ap.error("--heads applies to workloads without GQA")
        w["name"] = w["name"].replace(f"H={w['H']}", f"H={args.heads}")
        w["H"] = args.heads
    if args.oracle_sample_only:
        rate, dt, _ = oracle_sample(w, args.cpu_budget, learned=args.regime == "R2" and w.get("Hkv", w["H"]) == w["H"]
                                    and not w.get("lens"))
        print(json.dumps({"rate": rate, "seconds": dt}))
        return
    if args.train:
        out = run_train(args, w, rank, world) if args.impl == "ours" else None
        if out is not None and rank == 0:
            print(json.dumps(out))
        return
    if args.impl == "reference" and args.regime != "R2":
        ap.error("the reference arm times the oracle on the learned-selector workload only")
    out = run_reference(args, w, rank, world) if args.impl == "reference" else run_ours(args, w, rank, world)
    if out is not None and rank == 0:
        print(json.dumps(out))


if __name__ == "__main__":
    main()
