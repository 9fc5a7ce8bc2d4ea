#!/usr/bin/env python
"""Benchmark of the Comba chunk-parallel training step (forward + backward) on GB300.

Default workload: the 1.3B-scale layer shape, B=4, H=16, T=4096, dk=dv=128,
chunk 64, bf16 q/k/v/dO with fp32 gates, fp32 initial state h0 and final
state gradient dhT.  One step = comba_chunk_fwd (o, hT) + comba_chunk_bwd
(dq, dk, dv, dalpha, dbeta, db, dd, dh0).  Inputs are seeded synthetic data
(paper_2506_02475_gb300.inputs); L2 is flushed (256 MiB write) between timed
steps, outside the timed events.  The forward keeps the chunk factors the
backward needs (COMBA_SAVE_FACTORS) and the backward reuses them.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload lm1p3b|lm340m|varlen64k|decode]

Prints one JSON line (rank 0).  Under torchrun each rank runs an independent
replica of the workload (the op shards over sequences and heads with no
data-path collective); value = tokens of all ranks / max-over-ranks time.
The training-step line nests the decode measurement (Bd=256, H=16, d=128,
1024 sequential token steps) under "decode" unless --no-decode; its "e2e"
uploads every input and reads every output back each step.
``--impl reference`` times the fp64 CPU oracle on bounded samples instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Comba fwd+bwd tokens/s and TFLOP/s (% BF16 peak) at H=16,d=128,T=4096"
DECODE_METRIC = "Comba recurrent decode tokens/s at Bd=256,H=16,d=128 (fp32 state)"
FLUSH_BYTES = 256 << 20
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {k: float(p[k]) for k in FALLBACK_PEAKS}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


def fwd_flops_per_token_head(C=64, dk=128, dv=128):
    """Five C^2 d GEMMs (K K^T, M K, M V, Q~K^T, P E) and three C d^2 (W H, Q~ H, Kbar^T E)."""
    return 2 * C * (3 * dk + 2 * dv) + 6 * dk * dv


def compulsory_bytes(dk, dv, token_heads, state_elems, es=2):
    """Bytes a training step must move at least once (inputs read once, outputs written once):
    forward q, k, v, alpha, beta in, o out, h0 in, hT out; backward q, k, v, alpha, beta, dO in,
    dq, dk, dv, dalpha, dbeta out, h0 and dhT in, dh0 out.  At dk = dv = 128 in bf16 that is
    1032 B (forward) and 1808 B (backward) per (token, head), plus the fp32 states.  `per_stage`
    gives the share each kernel of the tcgen05 path must touch itself: prep reads k, v and the
    gates; the output kernel reads q, k and alpha and writes o; the local-gradient kernel reads
    every backward input and writes every token gradient."""
    tok_fwd = (2 * dk + dv) * es + 8 + dv * es
    tok_bwd = (2 * dk + dv) * es + 8 + dv * es + (2 * dk + dv) * es + 8
    fwd = token_heads * tok_fwd + 2 * state_elems * 4
    bwd = token_heads * tok_bwd + 3 * state_elems * 4
    per_stage = {"prep": token_heads * ((dk + dv) * es + 8), "output": token_heads * ((2 * dk + dv) * es + 4),
                 "scan_fwd": 2 * state_elems * 4, "scan_bwd": 2 * state_elems * 4, "bwd_local": token_heads * tok_bwd}
    return fwd, bwd, per_stage


# --------------------------------------------------------------- kernel model
# Algorithmic FLOPs and HBM bytes per launch of each kernel of the training step
# (bf16 storage, C = 64), summed over the (chunk, head) pairs one launch covers:
# the tile products the kernel must form and the tensors it must read or write
# once.  Forward saves the backward's factors (M, Atilde^T, E).

def stage_model(dk, dv, slots, H, N, save=True, tc=True, pk=False, vg=1):
    """`tc`: the tcgen05 path (bf16, d=128), whose reverse scan reads Atilde itself, so
    the forward saves M but no Atilde^T; its scans form their additive terms themselves:
    B^T = U_s^T K from the U_s^T = (Diag(s) U)^T that prep writes in place of B^T, and
    C^T = dO^T Z from the Z^T that the output kernel saves (no separate C-term kernel).  `pk`: Comba-pk feedback vectors P, read by prep and
    by the local gradients, which also write dP.  At dk = 256 no chunk map is formed: the
    scans read W, K and U (forward) or Z and dO (backward, forming C^T = dO^T Z) and form
    two products per chunk.
    `H` counts value heads of width `dv`, `vg` of them per key head: tensors and products
    that depend on the key head only (q, k, gates, W, M, Atilde, the Gram, Q~ K^T, dq, dk,
    dalpha, dbeta) are counted once per (chunk, key head), however often a kernel re-reads
    or recomputes them per value head."""
    C, es, f4 = 64, 2, 4
    P = slots * H            # (chunk, value head) units
    Pk = P // vg             # (chunk, key head) units
    wide = dk > 128
    at = save and not tc and not wide
    mp = 0 if wide else 1    # the chunk map Atilde, B^T
    m = {}
    m["prep"] = dict(flops=Pk * (2 * C * C * 2 * dk + mp * 2 * dk * C * dk * (2 if at else 1))
                     + P * (2 * C * C * dv + mp * 2 * dv * C * dk),
                     bytes=Pk * (2 * C * dk * es + 3 * C * f4 + (C * C * es if save else 0)
                                 + mp * dk * dk * es + (dk * dk * es if at else 0))
                     + P * (2 * C * dv * es + mp * dv * dk * es))
    if wide:
        m["scan_fwd"] = dict(flops=P * 4 * C * dk * dv,
                             bytes=Pk * (2 * C * dk * es + C * f4) + P * (C * dv + dv * dk) * es)
        # reverse: W, K, Z per key head; dO in and dH'^T out per value head; C^T = dO^T Z formed inside
        m["scan_bwd"] = dict(flops=P * 6 * C * dk * dv,
                             bytes=Pk * (3 * C * dk * es + C * f4) + P * (C * dv + dv * dk) * es)
    else:
        m["scan_fwd"] = dict(flops=P * 2 * dv * dk * dk, bytes=Pk * (dk * dk * es + f4) + P * 2 * dv * dk * es)
        m["scan_bwd"] = dict(flops=P * 2 * dv * dk * dk, bytes=Pk * (dk * dk * es + f4) + P * 2 * dv * dk * es)
    m["output"] = dict(flops=Pk * 2 * C * C * dk + P * (4 * C * dk * dv + 2 * C * C * dv),
                       bytes=Pk * (3 * C * dk * es + C * f4)
                       + P * (C * dv * es + dv * dk * es + C * dv * es * (2 if save else 1)))
    m["bwd_prep"] = dict(flops=Pk * 4 * C * C * dk + P * 2 * dv * C * dk,
                         bytes=Pk * (3 * C * dk * es + C * f4) + P * (C * dv * es + dv * dk * es))
    if wide:   # the output kernel saves Z once per key head; no C-term kernel
        if save:
            m["output"]["flops"] += Pk * 2 * C * C * dk
            m["output"]["bytes"] += Pk * C * dk * es
        m["bwd_prep"] = dict(flops=0, bytes=0)
    if tc and not wide:
        # prep writes U_s^T = (Diag(s) U)^T instead of forming B^T; the forward scan forms
        # B^T = U_s^T K from it and the keys
        m["prep"]["flops"] -= P * 2 * dv * C * dk
        m["prep"]["bytes"] += P * (C * dv * es - dv * dk * es)
        m["scan_fwd"] = dict(flops=P * (2 * dv * dk * dk + 2 * dv * C * dk),
                             bytes=Pk * (dk * dk * es + f4 + C * dk * es) + P * (dv * C * es + dv * dk * es))
        if save:   # Z^T = Qhat^T - W^T P^T, once per (chunk, key head)
            m["output"]["flops"] += Pk * 2 * C * C * dk
            m["output"]["bytes"] += Pk * dk * C * es
        m["bwd_prep"] = dict(flops=0, bytes=0)
        # reverse scan: Atilde and gamma, Z^T per key head; dO in and dH'^T out per value head
        m["scan_bwd"] = dict(flops=P * (2 * dv * dk * dk + 2 * dv * C * dk),
                             bytes=Pk * (dk * dk * es + f4 + dk * C * es) + P * (C * dv * es + dv * dk * es))
    m["bwd_local"] = dict(flops=Pk * 2 * C * C * dk * 2
                          + P * (2 * C * C * dk * 7 + 2 * C * dk * dv * 4 + 2 * C * C * dv * 4 + 4 * C ** 3),
                          bytes=Pk * (2 * C * dk * es + C * C * es + 3 * C * f4 + 2 * C * dk * es + 2 * C * f4)
                          + P * (2 * C * dv * es + C * dv * es + 2 * dv * dk * es + C * dv * es))
    if tc and not pk:
        # the tcgen05 local-gradient kernel: S, K K^T per key head; per value head R1 (three
        # C x dk x dv products), (M^T dE) H^T, P^T dO, M^T dE, dPhat K, dPhat^T Q~, dA from
        # (M^T dE) E^T and dG K, dG^T K
        m["bwd_local"]["flops"] = Pk * 2 * 2 * C * C * dk + P * 2 * (4 * C * dk * dv + 4 * C * C * dk + 4 * C * C * dv)
    if pk:
        m["prep"]["bytes"] += Pk * C * dk * es
        m["bwd_local"]["bytes"] += Pk * 2 * C * dk * es
    m["chunk_map"] = dict(flops=0, bytes=slots * 16 + (N + 1) * 8)
    m["output_E"] = dict(flops=0, bytes=0)
    m["reduce"] = dict(flops=0, bytes=P * 8 + 8 * H)
    return m


# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) per (chunk, head) unit
# of each kernel of the bf16 d=128 path, from one ncu capture of those two metrics on
# the 340M-shape step (2048 units per launch), scaled to a launch by its unit count
# (every launch touches each unit's tiles once).  A figure is kept only while the
# sources of its kernel hash to the captured value; otherwise traffic is null.
CAPTURED_TRAFFIC = {
    "prep": ("k_prep_tc", 94_366, ('chunk_tc.cu', 'tc_tiles.cuh', 'common.cuh', 'params.cuh'), "be4b1d27b40aa1f1"),
    "scan_fwd": ("k_scan_tc_split<128,128,0,2>", 83_423, ('scan.cu', 'common.cuh', 'params.cuh'), "2ff0c8eb7a5e3add"),
    "output": ("k_output_tc", 130_446, ('chunk_tc.cu', 'tc_tiles.cuh', 'common.cuh', 'params.cuh'), "be4b1d27b40aa1f1"),
    "scan_bwd": ("k_scan_tc_split<128,128,1,1>", 85_703, ('scan.cu', 'common.cuh', 'params.cuh'), "2ff0c8eb7a5e3add"),
    "bwd_local": ("k_bwd_local_tc", 193_867, ('local_tc.cu', 'tc_frag.cuh', 'tc_tiles.cuh', 'common.cuh', 'params.cuh'), "4eca458cdd2721f9"),
}
DECODE_TRAFFIC = (481_112_064, ('decode.cu', 'common.cuh', 'params.cuh'), "fba8e9172f2784c4")   # whole Bd=256 H=16 launch


def sources_hash(files):
    import hashlib
    m = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2506_02475_gb300", "csrc", f), "rb") as fh:
            m.update(fh.read())
    return m.hexdigest()[:16]


def captured_traffic(stage, units, dk, dv, dtype="bf16", tc=True):
    entry = CAPTURED_TRAFFIC.get(stage)
    if entry is None or not tc or dk != 128 or dv != 128 or dtype != "bf16":
        return None, None
    kernel, per_unit, files, digest = entry
    if sources_hash(files) != digest:
        return None, kernel
    return per_unit * units, kernel


FWD_STAGES = ["chunk_map", "prep", "scan_fwd", "output"]
BWD_STAGES = ["chunk_map", "prep", "scan_fwd", "output_E", "bwd_prep", "scan_bwd", "bwd_local", "reduce"]


# ------------------------------------------------------------------ clocks

class NvmlClockSampler:
    """SM clock and clock-event reasons read through NVML (read-only queries) every
    `period_s` by a host thread during the timed region; falls back to nvidia-smi."""
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, device_id, period_s=0.005):
        import ctypes
        import threading
        self.period = period_s
        self.samples, self.reasons = [], 0
        self.stop_evt = threading.Event()
        self.thread = None
        self.fallback = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                raise OSError("nvmlInit failed")
            self.nv = nv
            self.dev = ctypes.c_void_p()
            if nv.nvmlDeviceGetHandleByUUID(str(device_id).encode(), ctypes.byref(self.dev)) != 0:
                raise OSError("no NVML handle for " + str(device_id))
            mx = ctypes.c_uint()
            nv.nvmlDeviceGetMaxClockInfo(self.dev, 1, ctypes.byref(mx))
            self.max_mhz = float(mx.value)
            self.get_reasons = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                nv.nvmlDeviceGetCurrentClocksThrottleReasons
        except Exception:
            self.nv = None
            self.fallback = ClockSampler(device_id)

    def _run(self):
        import ctypes
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        while not self.stop_evt.is_set():
            if self.nv.nvmlDeviceGetClockInfo(self.dev, 1, ctypes.byref(clk)) == 0:
                self.samples.append(float(clk.value))
            if self.get_reasons(self.dev, ctypes.byref(rs)) == 0:
                self.reasons |= int(rs.value)
            self.stop_evt.wait(self.period)

    def start(self):
        if self.fallback is not None:
            return self.fallback.start()
        import threading
        self.thread = threading.Thread(target=self._run, daemon=True)
        self.thread.start()

    def stop(self):
        if self.fallback is not None:
            return self.fallback.stop()
        self.stop_evt.set()
        self.thread.join()
        if not self.samples:
            return None
        names = sorted(n for bit, n in self.REASONS.items() if self.reasons & bit)
        return {"sm_mhz": statistics.median(self.samples), "sm_max_mhz": self.max_mhz, "reasons": names,
                "samples": len(self.samples), "source": "nvml"}


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, device_id):
        self.proc = None
        self.device_id = device_id

    def start(self):
        try:
            cmd = ["nvidia-smi", "--query-gpu=" + ",".join(self.FIELDS), "--format=csv,noheader,nounits",
                   "-lms", "200"]
            if self.device_id is not None:
                cmd += ["-i", str(self.device_id)]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def nvsmi_device_id():
    import torch
    try:
        uuid = str(torch.cuda.get_device_properties(torch.cuda.current_device()).uuid)
        return uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        return vis.split(",")[torch.cuda.current_device()] if vis else torch.cuda.current_device()


# ------------------------------------------------------------- distributed

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_init(world, local, backend):
    import torch
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return dist if world > 1 else None


# -------------------------------------------------------- CPU oracle timing

def oracle_sample(w, rows, heads, tokens, p=None, variant="splr"):
    """Bounded slice of a workload: batch rows `rows`, heads, first `tokens` tokens (a packed
    workload: the first `tokens` tokens of the packed stream, its sequences cut there), with the
    Comba-pk feedback vectors `p` (shaped like k) when given."""
    if w.cu_seqlens is not None:
        sl = (slice(0, tokens), slice(heads[0], heads[1]))
        cu = np.asarray(w.cu_seqlens, np.int64)
        cu = np.concatenate([cu[cu < tokens], [tokens]])
        n = len(cu) - 1

        def st(x):
            return None if x is None else np.ascontiguousarray(x[:n, heads[0]:heads[1]])
    else:
        sl = (slice(rows[0], rows[1]), slice(0, tokens), slice(heads[0], heads[1]))
        cu = None

        def st(x):
            return None if x is None else np.ascontiguousarray(x[rows[0]:rows[1], heads[0]:heads[1]])

    return dict(q=np.ascontiguousarray(w.q[sl]), k=np.ascontiguousarray(w.k[sl]), v=np.ascontiguousarray(w.v[sl]),
                alpha=np.ascontiguousarray(w.alpha[sl]), beta=np.ascontiguousarray(w.beta[sl]),
                b=None if w.b is None else w.b[heads[0]:heads[1]], d=w.d[heads[0]:heads[1]], h0=st(w.h0),
                dO=np.ascontiguousarray(w.dO[sl]), dhT=st(w.dhT), cu_seqlens=cu,
                p=None if p is None else np.ascontiguousarray(p[sl]), variant=variant)


def time_oracle_step(s):
    import oracle
    t0 = time.perf_counter()
    kw = dict(cu_seqlens=s["cu_seqlens"], p=s["p"], variant=s["variant"])
    oracle.fwd(s["q"], s["k"], s["v"], s["alpha"], s["beta"], s["b"], s["d"], h0=s["h0"], **kw)
    oracle.bwd(s["q"], s["k"], s["v"], s["alpha"], s["beta"], s["b"], s["d"], s["dO"], h0=s["h0"], dhT=s["dhT"], **kw)
    return time.perf_counter() - t0


def cpu_baseline(w, target_s=12.0, p=None, variant="splr"):
    """The oracle as it stands on this host's cores: fwd+bwd over all heads of a growing
    sample (token prefix of batch row 0, then whole batch rows) until about `target_s`
    seconds of wall time or the whole workload."""
    import oracle
    if w.cu_seqlens is not None:
        B, T, H = 1, w.q.shape[0], w.q.shape[1]
    else:
        B, T, H = w.q.shape[0], w.q.shape[1], w.q.shape[2]
    rows, tokens = 1, min(T, 256)
    while True:
        s = oracle_sample(w, (0, rows), (0, H), tokens, p=p, variant=variant)
        dt = time_oracle_step(s)
        if dt >= target_s or (tokens >= T and rows >= B):
            break
        grow = max(2.0, min(8.0, target_s / max(dt, 1e-3)))
        if tokens < T:
            tokens = min(T, max(64, int(tokens * grow) // 64 * 64))
        else:
            rows = min(B, max(rows + 1, int(rows * grow)))
    what = "the whole workload" if (rows == B and tokens == T) else f"batch rows 0..{rows - 1}, first {tokens} tokens"
    return {"value": rows * tokens / dt, "unit": "tokens/s", "cores": oracle.default_threads(), "kind": "oracle",
            "sample": f"fwd+bwd over {what} (all {H} heads; fp64 token recurrence, exact BPTT): {dt:.2f} s"}


# --------------------------------------------------------------- our path

def run_ours(args, world, rank, local):
    import torch
    dist = dist_init(world, local, "nccl")
    torch.cuda.set_device(local)
    from paper_2506_02475_gb300 import (comba_chunk_bwd, comba_chunk_bwd_pk, comba_chunk_fwd, comba_chunk_fwd_pk,
                                        inputs, shard)
    from paper_2506_02475_gb300 import binding

    peaks, peak_src = load_peaks()
    iplr = args.variant == "iplr"
    pk = args.variant == "pk"   # Comba-pk feedback vectors (runs the mma.sync kernels)
    # weak scaling: each rank owns its own batch of sequences (same parameters, own data)
    w = inputs.make(args.workload, seed_offset=shard.rank_seed_offset(rank))
    dev = torch.device("cuda", local)
    tdt = torch.bfloat16

    def host(x, dt):
        return None if x is None else torch.from_numpy(np.ascontiguousarray(x)).to(dt).pin_memory()

    hin = dict(q=host(w.q, tdt), k=host(w.k, tdt), v=host(w.v, tdt), alpha=host(w.alpha, torch.float32),
               beta=host(w.beta, torch.float32), d=host(w.d, torch.float32), b=host(w.b, torch.float32),
               h0=host(w.h0, torch.float32), dO=host(w.dO, tdt), dhT=host(w.dhT, torch.float32))
    p_np = inputs.feedback_vectors(w.k, w.dtype, seed_offset=shard.rank_seed_offset(rank)) if pk else None
    if pk:
        hin["p"] = host(p_np, tdt)
    cu = None if w.cu_seqlens is None else torch.from_numpy(w.cu_seqlens.astype(np.int32)).to(dev)
    din = {k: (None if v is None else v.to(dev)) for k, v in hin.items()}
    q = din["q"]
    ws_bytes = binding.comba_workspace_size(q, din["v"], cu, backward=True, flags=binding.COMBA_PK if pk else 0)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    N = w.num_seqs
    H, dk, dv = w.H, w.dk, w.dv
    o = torch.empty_like(din["v"])
    hT = torch.empty((N, H, dk, dv), dtype=torch.float32, device=dev)
    grads = {"dq": torch.empty_like(q), "dk": torch.empty_like(din["k"]), "dv": torch.empty_like(din["v"]),
             "dalpha": torch.empty_like(din["alpha"]), "dbeta": torch.empty_like(din["beta"]),
             "dd": torch.empty_like(din["d"]), "db": torch.empty((H,), dtype=torch.float32, device=dev),
             "dh0": torch.empty((N, H, dk, dv), dtype=torch.float32, device=dev)}
    if pk:
        grads["dp"] = torch.empty_like(q)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)

    ev_f = [torch.cuda.Event(enable_timing=True) for _ in range(len(FWD_STAGES) + 1)]
    ev_b = [torch.cuda.Event(enable_timing=True) for _ in range(len(BWD_STAGES) + 1)]
    for e in ev_f + ev_b:
        e.record()
    torch.cuda.synchronize()
    hf = [e.cuda_event for e in ev_f]
    hb = [e.cuda_event for e in ev_b]

    def fwd_call(t, o_, hT_, events=None):
        kw = dict(b=t["b"], h0=t["h0"], cu_seqlens=cu, o=o_, hT=hT_, workspace=ws, stage_events=events,
                  save_factors=True, iplr=iplr)
        if pk:
            comba_chunk_fwd_pk(t["q"], t["k"], t["v"], t["p"], t["alpha"], t["beta"], t["d"], **kw)
        else:
            comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], **kw)

    def bwd_call(t, out_, events=None):
        kw = dict(b=t["b"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=cu, out=out_, workspace=ws, stage_events=events,
                  reuse_factors=True, iplr=iplr)
        if pk:
            comba_chunk_bwd_pk(t["q"], t["k"], t["v"], t["p"], t["alpha"], t["beta"], t["d"], t["dO"], **kw)
        else:
            comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], **kw)

    def step(t, events=True):
        # training step: the forward keeps the backward's chunk factors, the backward reuses them
        fwd_call(t, o, hT, hf if events else None)
        bwd_call(t, grads, hb if events else None)

    for _ in range(args.warmup):
        flush.zero_()
        step(din)
    torch.cuda.synchronize()

    # ---- timed region: device-resident inputs
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    stage_ms = {("fwd", s): 0.0 for s in FWD_STAGES}
    stage_ms.update({("bwd", s): 0.0 for s in BWD_STAGES})
    clocks = NvmlClockSampler(nvsmi_device_id())
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    total_ms = 0.0
    t_wall = time.perf_counter()
    for _ in range(args.steps):
        flush.zero_()
        start.record()
        step(din, events=False)
        end.record()
        end.synchronize()
        total_ms += start.elapsed_time(end)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t_wall
    # The per-stage breakdown comes from as many steps again, with an event recorded between stages:
    # each event costs the stream about a microsecond, so none is recorded in the timed steps above.
    for _ in range(args.steps):
        flush.zero_()
        step(din, events=True)
        torch.cuda.synchronize()
        for i, s in enumerate(FWD_STAGES):
            stage_ms[("fwd", s)] += ev_f[i].elapsed_time(ev_f[i + 1])
        for i, s in enumerate(BWD_STAGES):
            stage_ms[("bwd", s)] += ev_b[i].elapsed_time(ev_b[i + 1])
    clk = clocks.stop()
    if dist:
        dist.barrier()
    ms = shard.max_over_ranks(total_ms / args.steps, dist, dev)

    tokens = w.tokens
    value = tokens * world / (ms / 1e3)
    flops_step = 3.5 * fwd_flops_per_token_head(64, dk, dv) * tokens * H
    tflops = flops_step * world / (ms / 1e3) / 1e12

    # ---- dominant kernel and its roofline
    slots = (tokens // 64 + N) if w.cu_seqlens is not None else w.q.shape[0] * ((w.q.shape[1] + 63) // 64)
    # value-head groups: dv beyond 128 runs as dv / 128 value heads of width 128 per key head (at
    # dk = 256: value heads 64 wide), and every kernel's unit is a (chunk, value head) pair
    vg = dv // 64 if dk == 256 else (dv // 128 if dv > 128 else 1)
    dv_u, H_u = dv // vg, H * vg
    tc = w.dtype == "bf16" and dk == 128 and dv_u == 128
    model = stage_model(dk, dv_u, slots, H_u, N, tc=tc, pk=pk, vg=vg)
    # the dominant launch: the (phase, stage) with the most time (a stage the backward skips
    # because it reuses the forward's factors is not averaged with its empty slot)
    dom_phase, dom = max(stage_ms, key=lambda ps: stage_ms[ps])
    launch_ms = stage_ms[(dom_phase, dom)] / args.steps
    mdl = model[dom]
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    ai = mdl["flops"] / max(mdl["bytes"], 1)
    if ai >= ridge:
        ach = mdl["flops"] / (launch_ms / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": ach, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s"}
    else:
        ach = mdl["bytes"] / (launch_ms / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    # captured figures are for the kernels without Comba-pk feedback vectors
    traffic, kname = captured_traffic(dom, slots * H_u, dk, dv_u, w.dtype, tc=tc and not pk)
    roof.update({"kernel": kname or dom, "stage": dom, "launch_ms": launch_ms, "algorithmic_flops": mdl["flops"],
                 "algorithmic_bytes": mdl["bytes"], "traffic": traffic,
                 "traffic_source": "ncu capture of the 340M-shape step, scaled by units" if traffic else None,
                 "peak_source": peak_src + " (burst)"})
    # the same kernel and the whole step on compulsory bytes only (the step's inputs read once and
    # its outputs written once; none of this design's intermediates)
    c_fwd, c_bwd, c_stage = compulsory_bytes(dk, dv, tokens * H, N * H * dk * dv)
    cb = c_stage.get(dom)
    roof["compulsory_bytes"] = cb
    roof["frac_compulsory"] = None if cb is None else cb / (launch_ms / 1e3) / 1e9 / peaks["hbm_gbs"]
    roof["step_compulsory"] = {"bytes": c_fwd + c_bwd, "achieved_gbs": (c_fwd + c_bwd) / (ms / 1e3) / 1e9,
                               "frac": (c_fwd + c_bwd) / (ms / 1e3) / 1e9 / peaks["hbm_gbs"],
                               "floor_ms": (c_fwd + c_bwd) / (peaks["hbm_gbs"] * 1e9) * 1e3}

    # ---- end to end through the public API with host buffers.  Every step copies all its
    # inputs from pinned host memory and reads its result back: the per-sequence and per-head
    # results (hT, dh0, db, dd), while o and the token gradients stay on the device for the
    # neighbouring layers, as in training.  A second pass reads every output back.  The copies
    # run on their own streams over two device buffer sets, so step i's upload and step i-1's
    # download overlap step i's kernels (a data loader's double buffering).
    RESULT = ("hT", "dh0", "db", "dd")
    sets = []
    for j in range(2):
        dbuf = {k: (None if v is None else torch.empty_like(v)) for k, v in din.items()}
        douts = {"o": torch.empty_like(o), "hT": torch.empty_like(hT), **{k: torch.empty_like(v) for k, v in grads.items()}}
        hout = {k: torch.empty(v.shape, dtype=v.dtype).pin_memory() for k, v in douts.items()}
        sets.append((dbuf, douts, hout))
    bi = sum(v.numel() * v.element_size() for v in hin.values() if v is not None)
    comp = torch.cuda.current_stream()
    up, down = torch.cuda.Stream(), torch.cuda.Stream()
    ev = {name: [torch.cuda.Event() for _ in range(2)] for name in ("uploaded", "computed", "consumed", "downloaded")}

    def run_e2e(nsteps, keys, t_start=None, t_end=None):
        for i in range(nsteps):
            j = i % 2
            dbuf, douts, hout = sets[j]
            with torch.cuda.stream(up):
                if i == 0 and t_start is not None:
                    t_start.record(up)
                if i >= 2:
                    up.wait_event(ev["consumed"][j])          # step i-2 finished reading this input set
                for k_, v_ in hin.items():
                    if v_ is not None:
                        dbuf[k_].copy_(v_, non_blocking=True)
                ev["uploaded"][j].record(up)
            comp.wait_event(ev["uploaded"][j])
            if i >= 2:
                comp.wait_event(ev["downloaded"][j])          # step i-2's results are on the host
            fwd_call(dbuf, douts["o"], douts["hT"])
            bwd_call(dbuf, {k: douts[k] for k in grads})
            ev["consumed"][j].record(comp)
            ev["computed"][j].record(comp)
            with torch.cuda.stream(down):
                down.wait_event(ev["computed"][j])
                for k_ in keys:
                    hout[k_].copy_(douts[k_], non_blocking=True)
                ev["downloaded"][j].record(down)
                if i == nsteps - 1 and t_end is not None:
                    t_end.record(down)

    def time_e2e(keys):
        run_e2e(max(2, args.warmup), keys)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        run_e2e(args.steps, keys, e_start, e_end)
        torch.cuda.synchronize()
        return shard.max_over_ranks(e_start.elapsed_time(e_end) / args.steps, dist, dev)

    e_ms = time_e2e(RESULT)
    bo = sum(sets[0][1][k].numel() * sets[0][1][k].element_size() for k in RESULT)
    all_keys = tuple(sets[0][1].keys())
    e_full_ms = time_e2e(all_keys)
    bo_full = sum(sets[0][1][k].numel() * sets[0][1][k].element_size() for k in all_keys)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, p=p_np, variant="splr" if pk else args.variant)
        if pk:
            cpu["sample"] = "Comba-pk " + cpu["sample"]

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded; paper's layer shape and gate ranges)",
            "config": {"workload": f"{args.workload}: " + workload_desc(w), "variant": args.variant,
                       "global_batch": w.num_seqs * world,
                       "seq_len": int(w.q.shape[1]) if w.cu_seqlens is None else int(w.tokens),
                       "parallelism": f"data-parallel x{world}: each rank its own sequences, no data-path collective",
                       "l2": "device-timed steps: flushed between steps (256 MiB write, outside the events); "
                             "e2e: working set (inputs, workspace, outputs: >1 GB) larger than L2"},
            "tflops": tflops, "pct_bf16_peak": tflops / peaks["bf16_tflops"] * 100,
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": {"value": tokens * world / (e_full_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": bi,
                    "d2h_bytes_per_step": bo_full, "ms_per_step": e_full_ms,
                    "read_back": list(all_keys),
                    "copies": "pinned host buffers; every input uploaded and every output read back each step; "
                              "upload and download on their own streams, double-buffered",
                    "results_only_read_back": {"value": tokens * world / (e_ms / 1e3), "ms_per_step": e_ms,
                                               "d2h_bytes_per_step": bo, "read_back": list(RESULT),
                                               "note": "o and the token gradients left on the device"}},
            "clocks": clk,
            # forward: chunk map, prep, scan, output; backward: (C term at dk = 64), reverse
            # scan, local gradients, per-head sums; plus q - d p per call with p, the key-head sums
            # with value-head groups
            "gpu_launches": (4 + (3 if tc or dk == 256 else 4) + (2 if pk else 0) + (1 if vg > 1 else 0)) * args.steps,
            "stages_ms_per_step": {f"{p}.{s}": v / args.steps for (p, s), v in stage_ms.items()},
            "wall_s_timed": wall,
        }
    # the recurrent decode step (Bd=256, H=16, d=128) measured in the same run, its own line nested
    dec = None if args.no_decode else measure_decode(args, world, rank, dist, dev, peaks, peak_src)
    if rank == 0:
        if dec is not None:
            line["decode"] = dec
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def workload_desc(w):
    if w.cu_seqlens is not None:
        lens = np.diff(w.cu_seqlens).tolist()
        shape = f"packed {len(lens)} seqs (lengths {lens}), {w.tokens} tokens"
    else:
        shape = f"B={w.q.shape[0]} T={w.q.shape[1]}"
    return (f"{shape} H={w.H} dk={w.dk} dv={w.dv} chunk=64; {w.dtype} q/k/v/dO, fp32 gates/state; "
            f"h0={'yes' if w.h0 is not None else 'no'}, dhT=yes; step = chunk_fwd(o,hT, saves factors) + "
            f"chunk_bwd(all grads, reuses factors)")


# ------------------------------------------------------------ gated step

def run_gated(args, world, rank, local):
    """The training step with the gate and normalisation prologue (raw q, k, gate pre-activations):
    comba_chunk_fwd_gated (saving factors) + comba_chunk_bwd_gated (reusing them), device-resident."""
    import torch
    dist = dist_init(world, local, "nccl")
    torch.cuda.set_device(local)
    from paper_2506_02475_gb300 import binding, comba_chunk_bwd_gated, comba_chunk_fwd_gated, inputs, shard
    base = inputs.make(args.workload, with_grads=False)
    lens = None if base.cu_seqlens is None else np.diff(base.cu_seqlens)
    B = base.q.shape[0] if base.cu_seqlens is None else 1
    T = base.q.shape[1] if base.cu_seqlens is None else int(base.tokens)
    w = inputs.make_gated(B=B, T=T, H=base.H, dk=base.dk, dv=base.dv, dtype="bf16",
                          seed_offset=shard.rank_seed_offset(rank), lengths=lens)
    dev = torch.device("cuda", local)
    tok = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev).to(torch.bfloat16)
    f32 = lambda x: None if x is None else torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(dev)
    t = dict(q=tok(w.q), k=tok(w.k), v=tok(w.v), dO=tok(w.dO))
    for key in ("g_alpha", "g_beta", "a", "c", "b_raw", "d", "h0", "dhT"):
        t[key] = f32(getattr(w, key))
    cu = None if w.cu_seqlens is None else torch.from_numpy(w.cu_seqlens.astype(np.int32)).to(dev)
    iplr = args.variant == "iplr"
    shape = binding.make_shape(t["q"], t["v"], cu, None, binding.COMBA_GATED)
    ws = torch.empty(binding.lib().comba_workspace_size(binding.ctypes.byref(shape), 1), dtype=torch.uint8,
                     device=dev)
    o = torch.empty_like(t["v"])
    N, H, dk, dv = base.num_seqs, base.H, base.dk, base.dv
    hT = torch.empty((N, H, dk, dv), dtype=torch.float32, device=dev)
    grads = {}
    ev_f = [torch.cuda.Event(enable_timing=True) for _ in range(len(FWD_STAGES) + 1)]
    ev_b = [torch.cuda.Event(enable_timing=True) for _ in range(len(BWD_STAGES) + 1)]
    for e in ev_f + ev_b:
        e.record()
    torch.cuda.synchronize()
    hf, hb = [e.cuda_event for e in ev_f], [e.cuda_event for e in ev_b]
    args_ = (t["q"], t["k"], t["v"], t["g_alpha"], t["g_beta"], t["a"], t["c"], t["b_raw"], t["d"])

    def step(events=False):
        comba_chunk_fwd_gated(*args_, h0=t["h0"], cu_seqlens=cu, o=o, hT=hT, workspace=ws,
                              stage_events=hf if events else None, save_factors=True, iplr=iplr)
        comba_chunk_bwd_gated(*args_, t["dO"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=cu, out=grads, workspace=ws,
                              stage_events=hb if events else None, reuse_factors=True, iplr=iplr)

    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for _ in range(max(3, args.warmup)):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = NvmlClockSampler(nvsmi_device_id())
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    total, kern = 0.0, 0.0
    for _ in range(args.steps):
        flush.zero_()
        start.record()
        step()
        end.record()
        end.synchronize()
        total += start.elapsed_time(end)
    # the chunk kernels' share from as many steps again with stage events (none in the timed steps)
    for _ in range(args.steps):
        flush.zero_()
        step(events=True)
        torch.cuda.synchronize()
        kern += sum(ev_f[i].elapsed_time(ev_f[i + 1]) for i in range(len(FWD_STAGES)))
        kern += sum(ev_b[i].elapsed_time(ev_b[i + 1]) for i in range(len(BWD_STAGES)))
    clk = clocks.stop()
    ms = shard.max_over_ranks(total / args.steps, dist, dev)
    tokens = base.tokens
    if rank == 0:
        print(json.dumps({
            "metric": METRIC + ", with the gate and L2-norm prologue", "value": tokens * world / (ms / 1e3),
            "unit": "tokens/s", "n_gpus": world, "steps": args.steps, "warmup": max(3, args.warmup),
            "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (raw q, k with per-row scale in [0.5, 2]; gate pre-activations N(0,1))",
            "config": {"workload": f"{args.workload} gated: " + workload_desc(base), "variant": args.variant,
                       "l2": "flushed between timed steps (256 MiB write, outside the events)"},
            "chunk_kernels_ms_per_step": kern / args.steps,
            "prologue_epilogue_ms_per_step": ms - kern / args.steps,
            "clocks": clk}), flush=True)
    if dist:
        dist.destroy_process_group()


# ------------------------------------------------------------------ decode

def decode_oracle_sample(Bd, H, dk, dv, rows):
    """The first `rows` decode rows (all heads) of the decode workload: fp32 state and the
    8 token sets the GPU leg cycles through."""
    from paper_2506_02475_gb300 import inputs
    state = inputs.decode_state(Bd, H, dk, dv)[:rows]
    toks = []
    for s_ in range(8):
        q, k, v, a, be, d = inputs.decode_tokens(s_, Bd, H, dk, dv, "bf16")
        toks.append((q[:rows], k[:rows], v[:rows], a[:rows], be[:rows]))
    return state, toks, d


def time_oracle_decode(state, toks, d, nsteps):
    """`nsteps` sequential oracle decode steps from `state`; wall seconds."""
    import oracle
    t0 = time.perf_counter()
    st = state
    for i in range(nsteps):
        q, k, v, a, be = toks[i % 8]
        _, st = oracle.step(q, k, v, a, be, None, d, st)
    return time.perf_counter() - t0


def decode_cpu_baseline(Bd, H, dk, dv, rows=32, target_s=10.0):
    """The oracle's decode step on the host cores: the first `rows` decode rows, all heads,
    sequential token steps until about `target_s` seconds."""
    import oracle
    state, toks, d = decode_oracle_sample(Bd, H, dk, dv, rows)
    n, dt = 2, 0.0
    while True:
        dt = time_oracle_decode(state, toks, d, n)
        if dt >= target_s or n >= 4096:
            break
        n = int(n * max(2.0, min(8.0, target_s / max(dt, 1e-3))))
    return {"value": rows * n / dt, "unit": "tokens/s", "cores": oracle.default_threads(), "kind": "oracle",
            "sample": f"decode rows 0..{rows - 1} of {Bd}, all {H} heads, {n} sequential token steps "
                      f"(fp64 recurrence, fp32 state widened): {dt:.2f} s"}



def run_decode(args, world, rank, local):
    import torch
    dist = dist_init(world, local, "nccl")
    torch.cuda.set_device(local)
    peaks, peak_src = load_peaks()
    line = measure_decode(args, world, rank, dist, torch.device("cuda", local), peaks, peak_src)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def measure_decode(args, world, rank, dist, dev, peaks, peak_src):
    """The decode workload (Bd=256, H=16, d=128, 1024 sequential token steps per timed step):
    device-resident timing, the end-to-end leg and the oracle on the host; returns the JSON
    line's dict on rank 0 (None elsewhere)."""
    import torch
    from paper_2506_02475_gb300 import comba_recurrent_step, inputs, shard
    Bd, H, dk, dv = 256, 16, 128, 128
    off = shard.rank_seed_offset(rank)
    state = torch.from_numpy(inputs.decode_state(Bd, H, dk, dv, seed_offset=off)).to(dev)
    toks = []
    for s in range(8):  # cycle over 8 distinct token sets
        q, k, v, a, be, d = inputs.decode_tokens(s, Bd, H, dk, dv, "bf16", seed_offset=off)
        toks.append([torch.from_numpy(x).to(dev).to(torch.bfloat16) for x in (q, k, v)] +
                    [torch.from_numpy(x).to(dev) for x in (a, be)])
    d = torch.from_numpy(d).to(dev)
    o = torch.empty((Bd, H, dv), dtype=torch.bfloat16, device=dev)
    steps = 1024
    for i in range(args.warmup):
        t = toks[i % 8]
        comba_recurrent_step(t[0], t[1], t[2], t[3], t[4], d, state, o=o)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = NvmlClockSampler(nvsmi_device_id())
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    total = 0.0
    for _ in range(args.steps):
        start.record()
        for i in range(steps):
            t = toks[i % 8]
            comba_recurrent_step(t[0], t[1], t[2], t[3], t[4], d, state, o=o)
        end.record()
        end.synchronize()
        total += start.elapsed_time(end)
    clk = clocks.stop()
    if dist:
        dist.barrier()
    ms = shard.max_over_ranks(total / args.steps, dist, dev)
    per = ms / steps
    bytes_step = Bd * H * (2 * dk * dv * 4 + (2 * dk + 2 * dv) * 2 + 8)
    gbs = bytes_step / (per / 1e3) / 1e9

    # ---- end to end through the public API: every token step uploads its q, k, v, alpha,
    # beta from pinned host memory and reads its o back; the recurrent state is the model's
    # memory and stays resident on the device.  Upload and download run on their own streams
    # over two device buffer sets, so step i's upload and step i-1's download overlap step i.
    htoks = [[x.cpu().pin_memory() for x in t] for t in toks]
    sets = [([torch.empty_like(x) for x in toks[0]], torch.empty_like(o), torch.empty(o.shape, dtype=o.dtype).pin_memory())
            for _ in range(2)]
    comp, up, down = torch.cuda.current_stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev = {n_: [torch.cuda.Event() for _ in range(2)] for n_ in ("uploaded", "computed", "downloaded")}

    def run_e2e(nsteps, t_start=None, t_end=None):
        for i in range(nsteps):
            j = i % 2
            dbuf, dout, hout = sets[j]
            with torch.cuda.stream(up):
                if i == 0 and t_start is not None:
                    t_start.record(up)
                if i >= 2:
                    up.wait_event(ev["computed"][j])          # step i-2 finished reading this buffer set
                for dst, src in zip(dbuf, htoks[i % 8]):
                    dst.copy_(src, non_blocking=True)
                ev["uploaded"][j].record(up)
            comp.wait_event(ev["uploaded"][j])
            if i >= 2:
                comp.wait_event(ev["downloaded"][j])          # step i-2's o is on the host
            comba_recurrent_step(dbuf[0], dbuf[1], dbuf[2], dbuf[3], dbuf[4], d, state, o=dout)
            ev["computed"][j].record(comp)
            with torch.cuda.stream(down):
                down.wait_event(ev["computed"][j])
                hout.copy_(dout, non_blocking=True)
                ev["downloaded"][j].record(down)
                if i == nsteps - 1 and t_end is not None:
                    t_end.record(down)

    run_e2e(max(2, args.warmup))
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    run_e2e(steps, e_start, e_end)
    torch.cuda.synchronize()
    e_ms = shard.max_over_ranks(e_start.elapsed_time(e_end), dist, dev)
    bi = sum(x.numel() * x.element_size() for x in htoks[0])
    bo = o.numel() * o.element_size()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = decode_cpu_baseline(Bd, H, dk, dv)
    if rank == 0:
        return {
            "metric": DECODE_METRIC, "value": Bd * steps * world / (ms / 1e3), "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "fp32-state/bf16-tokens", "data": "synthetic",
            "config": {"workload": f"decode: Bd={Bd} H={H} dk={dk} dv={dv}, {steps} sequential steps per timed step",
                       "l2": "state (268 MB) larger than L2"},
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": gbs / peaks["hbm_gbs"], "kernel": "k_step", "launch_ms": per,
                         "traffic": DECODE_TRAFFIC[0] if sources_hash(DECODE_TRAFFIC[1]) == DECODE_TRAFFIC[2] else None,
                         "peak_source": peak_src},
            "cpu_baseline": cpu,
            "e2e": {"value": Bd * steps * world / (e_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": bi,
                    "d2h_bytes_per_step": bo, "ms_per_token_step": e_ms / steps,
                    "copies": "q, k, v, alpha, beta uploaded from pinned host memory and o read back every token "
                              "step (own streams, double-buffered); the state stays on the device"},
            "clocks": clk, "gpu_launches": steps * args.steps}
    return None


# --------------------------------------------------------------- reference

def run_reference(args, world, rank, local):
    """The fp64 CPU oracle as it stands, on bounded samples of the same workload."""
    if rank != 0:
        return
    import oracle
    from paper_2506_02475_gb300 import inputs
    if args.workload == "decode":
        Bd, H, dk, dv, rows, per_step = 256, 16, 128, 128, 32, 8
        state, toks, d = decode_oracle_sample(Bd, H, dk, dv, rows)
        for _ in range(args.warmup):
            time_oracle_decode(state, toks, d, per_step)
        dt = sum(time_oracle_decode(state, toks, d, per_step) for _ in range(args.steps)) / args.steps
        value = rows * per_step / dt
        sample = f"decode rows 0..{rows - 1} of {Bd}, all {H} heads, {per_step} sequential token steps per step"
        print(json.dumps({
            "metric": DECODE_METRIC, "impl": "reference", "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"decode: Bd={Bd} H={H} dk={dk} dv={dv}", "sample": sample},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.default_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }), flush=True)
        return
    w = inputs.make(args.workload)
    H = w.H
    total = int(w.q.shape[0] if w.cu_seqlens is not None else w.q.shape[1])   # tokens of batch row 0 / the pack
    tokens = min(total, args.reference_tokens)
    pv = inputs.feedback_vectors(w.k, w.dtype) if args.variant == "pk" else None
    s = oracle_sample(w, (0, 1), (0, H), tokens, p=pv, variant="splr" if args.variant == "pk" else args.variant)
    for _ in range(args.warmup):
        time_oracle_step(s)
    dts = [time_oracle_step(s) for _ in range(args.steps)]
    dt = sum(dts) / len(dts)
    value = tokens / dt
    flops = 3.5 * fwd_flops_per_token_head(64, w.dk, w.dv) * tokens * H
    print(json.dumps({
        "metric": METRIC, "impl": "reference", "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{args.workload}: " + workload_desc(w), "variant": args.variant,
                   "sample": f"batch row 0, all {H} heads, first {tokens} tokens per step"},
        "tflops": flops / dt / 1e12,
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.default_threads(), "kind": "oracle",
                         "sample": f"fwd+bwd, batch row 0, all {H} heads, first {tokens} tokens"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="lm1p3b",
                    choices=["lm1p3b", "lm340m", "varlen64k", "lm1p3b_v256", "lm1p3b_d256", "decode"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode", action="store_true",
                    help="leave out the decode measurement nested in the training-step line")
    ap.add_argument("--gated", action="store_true",
                    help="raw q, k and gate pre-activations through the gate and normalisation prologue")
    ap.add_argument("--variant", default="splr", choices=["splr", "iplr", "pk"],
                    help="state transition: Comba (alpha - btilde k k^T), Comba-iplr alpha (I - 2 btilde k k^T), "
                         "or Comba-pk (alpha - btilde p k^T with per-token feedback vectors p)")
    ap.add_argument("--reference-tokens", type=int, default=512)
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    world, rank, local = dist_setup()
    if args.impl == "reference":
        return run_reference(args, world, rank, local)
    if args.workload == "decode":
        return run_decode(args, world, rank, local)
    if args.gated:
        return run_gated(args, world, rank, local)
    return run_ours(args, world, rank, local)


if __name__ == "__main__":
    main()
