#!/usr/bin/env python
"""Benchmark of the triadic linear attention hot path on GB300.

A step is one chunkwise forward (saving what the backward needs) plus the
backward of triadic Gated DeltaNet on the headline workload (B=8, H=16, T=8192,
d_k=d_v=128, E=4, chunk 64, bf16 inputs / fp32 state), synthetic seeded
inputs.  The single-token decode step is measured in the same run on the
decode workload (fp32 state [256,32,8,128,128], 100 steps each of sGLA and
GDN after a 512-token chunked prefill) and reported under "decode", and the
same step with the headline's tokens packed into documents of log-normal length
around 1000 tokens (cu_seqlens, each document from its own state) under "packed";
the per-head-gate and E = 32 / d_k = 64 variants under "variants"; the layer's
fused input path and output gate (GB/s) under "layer_io"; the forward-only
workloads (GDN bf16 B=4 H=16 T=4096 E=8, long-context GDN B=1 H=32 T=65536
E=16, fp32 sGLA B=1 H=2 T=256 d=32 E=4) under "fwd_workloads".  Every call is
also set against the method's algorithmic flops and bytes ("s8d": the larger of
its tensor-core and HBM times at the measured peaks, as a fraction of the
measured time); the bytes this implementation moves are reported separately
("impl_bytes").

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (torchrun) every rank runs its own batch of independent sequences
(heads and sequences never interact): weak scaling, no collective on the data
path.  Rank 0 prints one JSON line.  `--impl reference` times the float64 CPU
oracle on this machine's host cores on a bounded sample of the same workload.
"""
import argparse
import ctypes
import dataclasses
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

import torch  # noqa: E402

HEADLINE_METRIC = "tokens/s triadic GDN fwd+bwd (T=8K, E=4); TFLOP/s and decode GB/s vs GB300 peak"
CHUNK = 64
OUT_DTYPE = torch.float32    # o, dq, dk, dv, dq', dk' (fp32, the accumulation precision); dg, dbeta fp32


def make_grads(x, out_dtype, dev):
    """Gradient buffers: dq, dk, dv, dq', dk' in out_dtype; dg and dbeta fp32."""
    od = dict(dtype=out_dtype, device=dev)
    return {"dq": torch.empty(x["q"].shape, **od), "dk": torch.empty(x["k"].shape, **od),
            "dv": torch.empty(x["v"].shape, **od), "dq2": torch.empty(x["q2"].shape, **od),
            "dk2": torch.empty(x["k2"].shape, **od),
            "dg": torch.empty(x["g"].shape, dtype=torch.float32, device=dev),
            "dbeta": torch.empty(x["beta"].shape, dtype=torch.float32, device=dev)}


# ----------------------------------------------------------------------------- helpers

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def rank_ops(ws_n, device):
    """barrier() and max_over_ranks(x) of a run with ws_n ranks.  With one rank both are no-ops;
    with more, a process-group barrier and an all-reduce MAX of one float64 on `device`: the
    run's only collectives, on timings, never on data (ranks process independent sequences)."""
    def barrier():
        if ws_n > 1:
            torch.distributed.barrier()

    def max_over_ranks(x):
        if ws_n == 1:
            return x
        t = torch.tensor([x], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        return float(t.item())

    return barrier, max_over_ranks


def job_tokens_per_s(ws_n, tokens_per_rank_step, ms_step_max):
    """Whole-job throughput under weak scaling: each of ws_n ranks processes its own
    tokens_per_rank_step per step, and the job's step takes the slowest rank's time."""
    return ws_n * tokens_per_rank_step / (ms_step_max / 1e3)


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def flops_per_token_head(kernel, E, dk, dv, C=CHUNK):
    """Algorithmic flops of one token of one head for each kernel (dense contractions).

    Forward recurrence: K S_e, Q S_e, K^T diag(w_e) U  -> 6 E dk dv; T Res, A U -> 4 C dv.
    Backward recurrence: K dS'_e, Q^T.., K^T..        -> 6 E dk dv; A^T dO, T^T dU -> 4 C dv.
    Chunk gradients: dO S^T, dRes S^T, U dS'^T        -> 6 E dk dv; dO U^T, dU Res^T -> 4 C dv;
                     Q K^T, K K^T, P K, P^T Q, (dKK+dKK^T) K -> 10 C dk; two C x C x C -> 4 C.
    Chunk prep: Q K^T, K K^T -> 4 C dk; triangular solve -> C^2/3.
    """
    name = kernel
    if name.startswith("fwd_recurrence") or name.startswith("bwd_recurrence"):
        return 6 * E * dk * dv + 4 * C * dv
    if name.startswith("bwd_chunk_grads"):
        return 6 * E * dk * dv + 4 * C * dv + 10 * C * dk + 4 * C
    if name.startswith("chunk_prep"):
        return 4 * C * dk + C * C / 3
    return 0.0


def bytes_per_token_head(kernel, E, dk, dv, C=CHUNK, in_b=2, out_b=4, delta=True, save=True):
    """Algorithmic HBM bytes of one token of one head for each kernel of the tensor-core path.

    Every tensor a kernel reads or writes is counted once (re-reads that the design leaves to
    L2, e.g. the key/query tiles shared by a head's value blocks, are not counted).  bf16
    hi/lo operands take 4 bytes per element; per-chunk matrices are divided by C tokens.
      gate cumsum:  log gates in, chunk-local cumsum out (fp32).
      chunk prep:   k, q, k', q', G, beta in; N (delta rule), [T; A T] and [A^T; T^T] hi/lo
                    tiles (2 x 128 x 64 and 4 x 64 x 64 bf16 per chunk), coefficient block out
                    (without a backward to follow, only [T; A T] and the coefficients).
      forward:      k, q, v, [T; A T], coefficients in; o, the chunk-start state checkpoint
                    (E dk dv hi/lo per chunk), U and Res token tiles out (without a backward
                    to follow, o alone).
      backward:     k, q, dO, [A^T; T^T], coefficients in; dv, the state-gradient checkpoint,
                    dU and -dRes token tiles out.
      gradients:    k, q, dO, U, Res, dU, -dRes, both checkpoints, N, G, k', q', beta in;
                    dq, dk, dq', dk', dg, dbeta out.
    """
    ck = E * dk * dv * 4 / C
    coef = (3 * C * E + 16) * 4 / C
    tiles = 8 * C                  # a 2 x 128 x 64 or 4 x 64 x 64 bf16 tile pair per chunk
    name = kernel
    if name.startswith("gate_cumsum"):
        return 8 * E
    if name.startswith("chunk_prep"):
        return ((2 * dk * in_b + 2 * E * in_b + 4 * E + 4) + (4 * C if delta and save else 0)
                + (2 if save else 1) * tiles + coef)
    if name.startswith("fwd_recurrence"):
        if not save:   # no checkpoints and no token tiles for a backward
            return (in_b * (2 * dk + dv) + tiles + coef) + dv * out_b
        return (in_b * (2 * dk + dv) + tiles + coef) + (dv * out_b + ck + 4 * dv * 2)
    if name.startswith("bwd_recurrence"):
        return (in_b * (2 * dk + dv) + tiles + coef) + (dv * out_b + ck + 4 * dv * (2 if delta else 1))
    if name.startswith("bwd_chunk_grads"):
        return (in_b * (2 * dk + dv) + 4 * dv * (4 if delta else 3) + 2 * ck + (4 * C if delta else 0)
                + 4 * E + 2 * E * in_b + 4) + (2 * dk * out_b + 2 * E * out_b + 4 * E + 4)
    return 0.0


def s8d_flops_per_token_head(E, dk, dv, backward, C=CHUNK):
    """Algorithmic flops of the method per token-head, counted on the chunk form (dense
    contractions only): forward 6 E dk dv + 4 C (dk + dv) + C^2 / 3 (state reads and update,
    the intra-chunk products, the triangular solve); forward + backward
    18 E dk dv + 12 C (dk + dv) (the backward doubles the forward's contractions)."""
    if backward:
        return 18 * E * dk * dv + 12 * C * (dk + dv)
    return 6 * E * dk * dv + 4 * C * (dk + dv) + C * C / 3


def s8d_bytes_per_token_head(E, dk, dv, backward, in_b=2, out_b=2, ckpt_b=2, C=CHUNK):
    """Algorithmic HBM bytes of the method per token-head: every input read once and every
    output written once (q, k, v, q', k' and o in bf16; log gates and beta fp32); with the
    backward also dO in and dq, dk, dv, dq', dk' (bf16), dg, dbeta (fp32) out, plus one bf16
    chunk-start state per chunk written by the forward and read by the backward."""
    inputs_b = in_b * (2 * dk + dv + 2 * E) + 4 * E + 4
    fwd = inputs_b + out_b * dv
    if not backward:
        return fwd
    bwd = inputs_b + in_b * dv + out_b * (2 * dk + dv + 2 * E) + 4 * E + 4
    return fwd + bwd + 2 * ckpt_b * E * dk * dv / C


def s8d_roofline(E, dk, dv, backward, units, ms, peaks):
    """The whole call against its algorithmic work: achieved TFLOP/s and GB/s, the fraction of
    the measured peaks, and the call's roofline time (the larger of the tensor and HBM times)."""
    f = s8d_flops_per_token_head(E, dk, dv, backward) * units
    b = s8d_bytes_per_token_head(E, dk, dv, backward) * units
    t_tc = f / (peaks["bf16_tflops_sustained"] * 1e12)
    t_hbm = b / (peaks["hbm_gbs"] * 1e9)
    s = ms / 1e3
    return {"flop": f, "bytes": b, "tflops": round(f / s / 1e12, 3),
            "tensor_frac": round(f / s / 1e12 / peaks["bf16_tflops_sustained"], 5),
            "gbs": round(b / s / 1e9, 1), "hbm_frac": round(b / s / 1e9 / peaks["hbm_gbs"], 5),
            "bound": "tensor" if t_tc >= t_hbm else "hbm",
            "roofline_ms": round(max(t_tc, t_hbm) * 1e3, 4),
            "frac": round(max(t_tc, t_hbm) / s, 5),
            "peaks": "bf16 dense sustained and HBM copy bandwidth, " + peaks["source"]}


def kernel_source_hash(kernel):
    """Hash of the source that builds a kernel: the .cu files that define it (`<name>_kernel`)
    and every local header they include, recursively (to invalidate stale ncu traffic)."""
    csrc = os.path.join(ROOT, "paper_2609_36529_gb300", "csrc")
    files, todo = set(), []
    for fn in sorted(os.listdir(csrc)):
        path = os.path.join(csrc, fn)
        if fn.endswith(".cu"):
            with open(path, "rb") as f:
                if (kernel + "_kernel").encode() in f.read():
                    todo.append(path)
    while todo:
        path = os.path.normpath(todo.pop())
        if path in files or not os.path.exists(path):
            continue
        files.add(path)
        with open(path) as f:
            for line in f:
                line = line.strip()
                if line.startswith("#include \""):
                    todo.append(os.path.join(os.path.dirname(path), line.split('"')[1]))
    h = hashlib.sha256()
    for path in sorted(files):
        h.update(os.path.relpath(path, ROOT).encode())
        with open(path, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic(kernel, units_per_launch):
    """DRAM bytes per launch from the committed ncu summary, if it is still current."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        rec = d[kernel]
        if rec.get("src_hash") != kernel_source_hash(kernel):
            return None
        return rec["bytes_per_unit"] * units_per_launch
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi samples (200 ms) of SM clock and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.samples = []
        self.proc = None
        self.thread = None
        sel = []
        try:
            uuid = str(torch.cuda.get_device_properties(device).uuid)
            sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            sel = []
        self.cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                    "-lms", "200"] + sel

    def _reader(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.samples.append(parts)

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
            self.thread = threading.Thread(target=self._reader, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        return self

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.thread.join(timeout=5)
        return self.summary()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]}
        sm, smax, power, reasons = [], [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for s in self.samples:
            try:
                sm.append(float(s[1]))
                smax.append(float(s[2]))
                power.append(float(s[3]))
            except ValueError:
                continue
            for name, val in zip(names, s[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        loaded = [x for x in sm if x > 0.5 * max(sm)] if sm else []
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def bad_clocks(c):
    if any(r in c.get("reasons", []) for r in ("hw_slowdown", "hw_thermal_slowdown",
                                                "sw_thermal_slowdown")):
        return True
    if c.get("sm_mhz") and c.get("sm_max_mhz") and c["sm_mhz"] < 0.6 * c["sm_max_mhz"] \
            and "sw_power_cap" not in c.get("reasons", []):
        return True
    return False


def profile_read(lib, stream):
    names = ctypes.create_string_buffer(64 * 32)
    launches = (ctypes.c_int * 32)()
    ms = (ctypes.c_float * 32)()
    n = lib.tla_profile_end(ctypes.c_void_p(stream), names, launches, ms, 32)
    if n < 0:
        raise RuntimeError(f"tla_profile_end failed: {n}")
    out = {}
    for i in range(n):
        nm = names.raw[64 * i:64 * (i + 1)].split(b"\0", 1)[0].decode()
        out[nm] = {"launches": int(launches[i]), "ms": float(ms[i])}
    return out


# ----------------------------------------------------------------------------- our arm

def run_ours(args):
    from paper_2609_36529_gb300 import inputs, tla

    ws_n, rank, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws_n > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    lib = tla.lib()
    lib.tla_profile_begin.restype = ctypes.c_int
    lib.tla_profile_end.argtypes = [ctypes.c_void_p, ctypes.c_char_p,
                                    ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_float),
                                    ctypes.c_int]
    lib.tla_profile_end.restype = ctypes.c_int

    barrier, max_over_ranks = rank_ops(ws_n, dev)

    w = inputs.GDN_FWDBWD_BF16
    if args.batch:   # profiling option: fewer sequences of the same shape
        w = dataclasses.replace(w, B=args.batch, name=f"{w.name}_batch{args.batch}")
    x = inputs.workload_inputs(w, device=dev, seed=rank)
    stream = torch.cuda.current_stream(dev)

    # preallocated outputs and workspaces (allocation is outside the timed region): o and every
    # gradient fp32 (the kernels accumulate in fp32; bf16 results are a variant below)
    o = torch.empty(w.B, w.T, w.H, w.dv, dtype=OUT_DTYPE, device=dev)
    p = tla.make_problem(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], None, o,
                         None, use_delta=True)
    fws = torch.empty(tla.fwd_workspace_bytes(p, True), dtype=torch.uint8, device=dev)
    bws = torch.empty(tla.bwd_workspace_bytes(p), dtype=torch.uint8, device=dev)
    grads = make_grads(x, OUT_DTYPE, dev)

    def step(xx):
        tla.tla_chunk_fwd(xx["q"], xx["k"], xx["v"], xx["q2"], xx["k2"], xx["g"], xx["beta"],
                          None, use_delta=True, save_for_bwd=True, want_ht=False, o=o,
                          workspace=fws)
        if args.fwd_only:
            return
        tla.tla_chunk_bwd(xx["q"], xx["k"], xx["v"], xx["q2"], xx["k2"], xx["g"], xx["dO"], fws,
                          beta=xx["beta"], use_delta=True, workspace=bws, grads=grads)

    for _ in range(args.warmup):
        step(x)
    torch.cuda.synchronize()
    if tla.tla_last_device_status() != 0:
        raise RuntimeError("device status not OK after warm-up")

    def timed_loop():
        barrier()
        torch.cuda.synchronize()
        clocks = ClockSampler(dev).start()
        time.sleep(0.25)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        lib.tla_profile_begin()
        e0.record(stream)
        for _ in range(args.steps):
            step(x)
        e1.record(stream)
        torch.cuda.synchronize()
        prof = profile_read(lib, stream.cuda_stream)
        barrier()
        ck = clocks.stop()
        return e0.elapsed_time(e1), prof, ck

    ms_total, prof, ck = timed_loop()
    remeasured = False
    if bad_clocks(ck):
        ms_total, prof, ck = timed_loop()
        remeasured = True
    ms_step = max_over_ranks(ms_total / args.steps)
    tokens_step = w.B * w.T
    value = job_tokens_per_s(ws_n, tokens_step, ms_step)
    if tla.tla_last_device_status() != 0:
        raise RuntimeError("device status not OK after timed loop")

    peaks = load_peaks()
    units = w.B * w.T * w.H  # token-heads per launch
    kernels = kernel_table(prof, w, units, peaks)
    top = max(prof, key=lambda n: prof[n]["ms"])
    top_avg_s = prof[top]["ms"] / prof[top]["launches"] / 1e3
    peak = peaks["bf16_tflops_sustained"]
    hbm = peaks["hbm_gbs"]
    # The dominant kernel against its share of the method's algorithmic flops (the chunk
    # kernels' work is dense contractions; its algorithmic bytes are far below its flops at
    # the measured peaks).  The bytes this design moves (bf16 hi/lo checkpoints and token
    # tiles, coefficient blocks) are reported beside it as impl_bytes, a different quantity.
    top_flops = flops_per_token_head(top, w.E, w.dk, w.dv) * units
    top_impl_bytes = bytes_per_token_head(top, w.E, w.dk, w.dv) * units
    achieved = top_flops / top_avg_s / 1e12
    roofline = {"kernel": top, "bound": "tensor", "achieved": round(achieved, 3), "peak": peak,
                "unit": "TFLOP/s", "frac": round(achieved / peak, 5),
                "traffic": ncu_traffic(top, units), "algorithmic_flops": int(top_flops),
                "avg_ms": round(top_avg_s * 1e3, 4),
                "peak_source": f"bf16 dense sustained, {peaks['source']} (MEASURED_PEAKS.json)"
                if peaks["source"] == "measured" else "bf16 dense sustained, fallback",
                "impl_bytes": int(top_impl_bytes),
                "impl_bytes_gbs": round(top_impl_bytes / top_avg_s / 1e9, 1),
                "impl_bytes_frac": round(top_impl_bytes / top_avg_s / 1e9 / hbm, 4)}
    total_flops = sum(flops_per_token_head(n, w.E, w.dk, w.dv) * units * prof[n]["launches"]
                      for n in prof) / args.steps
    total_bytes = sum(bytes_per_token_head(n, w.E, w.dk, w.dv) * units * prof[n]["launches"]
                      for n in prof) / args.steps
    step_s8d = s8d_roofline(w.E, w.dk, w.dv, True, units, ms_step, peaks)
    roofline["frac_s8d"] = step_s8d["frac"]
    gpu_launches = sum(r["launches"] for r in prof.values())

    # ---- end to end through the public API from pinned host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, tla, x, w, dev, stream, o, fws, bws, grads, barrier, max_over_ranks,
                      ws_n)

    # ---- the forward-only workloads (bf16 E=8 T=4096, long-context E=16 T=65536, fp32 sGLA)
    fwd_loads = None
    if not args.no_fwd_workloads:
        fwd_loads = run_fwd_workloads(args, tla, inputs, dev, stream, lib, peaks, barrier,
                                      max_over_ranks, ws_n, rank)
    packed = None
    if not args.no_packed:
        packed = run_packed(args, tla, inputs, w, dev, stream, barrier, max_over_ranks, ws_n, rank)
        packed["vs_uniform_batch"] = round(packed["value"] / value, 4)
    variants = None
    if not args.no_variants:
        variants = run_variants(args, tla, inputs, w, dev, stream, barrier, max_over_ranks, ws_n,
                                rank, value)
    layer = None
    if not args.no_layer:
        layer = run_layer_io(args, tla, inputs, w, dev, stream, barrier, max_over_ranks, rank,
                             load_peaks())
    decode = None
    if not args.no_decode:
        del fws, bws
        torch.cuda.empty_cache()
        decode = run_decode(args, tla, inputs, dev, stream, lib, peaks, barrier, max_over_ranks,
                            ws_n)

    # ---- CPU baseline: the oracle on this host's cores (rank 0, N=1 only)
    cpu = None
    if rank == 0 and ws_n == 1 and not args.no_cpu_baseline:
        cpu = oracle_baseline(x, w, seconds_target=args.cpu_seconds)

    if args.fwd_only or args.batch:
        print("bench: profiling options given; this line is not the headline measurement",
              file=sys.stderr)
    if rank == 0:
        line = {
            "metric": HEADLINE_METRIC, "value": round(value, 1), "unit": "tokens/s",
            "n_gpus": ws_n, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms_step, 4), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "T": w.T, "H": w.H, "dk": w.dk, "dv": w.dv,
                       "E": w.E, "chunk": CHUNK, "variant": "triadic GDN (joint-key delta rule)",
                       "state": "fp32", "outputs": "fp32 o and gradients",
                       "parallelism": f"replicas x{ws_n} (independent sequences)",
                       "l2": "inputs larger than L2 (q,k,v,dO 268 MB each per GPU)"},
            "tflops": round(total_flops / (ms_step / 1e3) / 1e12, 3),
            "tflops_frac": round(total_flops / (ms_step / 1e3) / 1e12 / peak, 5),
            "s8d": step_s8d,
            "step_impl_bytes": {"gb": round(total_bytes / 1e9, 3),
                                "achieved_gbs": round(total_bytes / (ms_step / 1e3) / 1e9, 1),
                                "frac": round(total_bytes / (ms_step / 1e3) / 1e9 / hbm, 4),
                                "note": "bytes this design moves (hi/lo checkpoints, token "
                                        "tiles, coefficient blocks), not the method's"},
            "roofline": roofline, "kernels": kernels, "gpu_launches": gpu_launches,
            "clocks": ck, "clocks_remeasured": remeasured,
            "e2e": e2e, "fwd_workloads": fwd_loads, "packed": packed, "variants": variants,
            "layer_io": layer, "decode": decode, "cpu_baseline": cpu, "impl": "ours",
        }
        print(json.dumps(line), flush=True)
    if ws_n > 1:
        torch.distributed.destroy_process_group()


def kernel_table(prof, w, units, peaks):
    """Per kernel of a profiled loop: launches, mean device time, share of the loop, achieved
    TFLOP/s on its algorithmic flops (fraction of the sustained bf16 peak) and the GB/s of the
    bytes this design moves through it (impl_gbs, fraction of the HBM copy bandwidth)."""
    tot = max(sum(v["ms"] for v in prof.values()), 1e-9)
    out = {}
    for name, r in prof.items():
        f = flops_per_token_head(name, w.E, w.dk, w.dv) * units
        by = bytes_per_token_head(name, w.E, w.dk, w.dv, delta=w.use_delta, save=w.backward) * units
        avg_s = r["ms"] / max(r["launches"], 1) / 1e3
        out[name] = {"launches": r["launches"], "avg_ms": round(avg_s * 1e3, 4),
                     "share": round(r["ms"] / tot, 4),
                     "tflops": round(f / avg_s / 1e12, 2) if f else None,
                     "tensor_frac": round(f / avg_s / 1e12 / peaks["bf16_tflops_sustained"], 4)
                     if f else None,
                     "impl_gbs": round(by / avg_s / 1e9, 1) if by else None,
                     "impl_hbm_frac": round(by / avg_s / 1e9 / peaks["hbm_gbs"], 4) if by else None}
    return out


def run_fwd_workloads(args, tla, inputs, dev, stream, lib, peaks, barrier, max_over_ranks, ws_n,
                      rank):
    """The forward-only workloads: triadic GDN forward bf16 B=4 H=16 T=4096 E=8 (zero initial
    state), the long-context forward B=1 H=32 T=65536 E=16 (initial state ~ N(0, 0.01)), both
    returning o (fp32) and the final state, and the fp32 sGLA forward B=1 H=2 T=256 d=32 E=4
    (latency-bound; time only).  Each: tokens/s, per-kernel shares from the library's own event
    timing, and the whole call against the algorithmic flops and bytes of the forward."""
    out = {}
    for w in (inputs.GDN_FWD_BF16, inputs.GDN_LONG_BF16, inputs.SGLA_FWD_FP32):
        x = inputs.workload_inputs(w, device=dev, seed=rank)
        o = torch.empty(w.B, w.T, w.H, w.dv, dtype=torch.float32, device=dev)
        ht = torch.empty(w.B, w.H, w.E, w.dk, w.dv, dtype=torch.float32, device=dev)
        p = tla.make_problem(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                             x["h0"], o, ht, use_delta=w.use_delta)
        fws = torch.empty(tla.fwd_workspace_bytes(p, False), dtype=torch.uint8, device=dev)

        def step():
            tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                              x["h0"], use_delta=w.use_delta, save_for_bwd=False, o=o, ht=ht,
                              workspace=fws)

        k = 20 if w.B * w.T <= 4096 else 5
        for _ in range(3):
            step()
        torch.cuda.synchronize()
        barrier()
        lib.tla_profile_begin()
        ms = _time_steps(step, k, 0, stream, barrier, max_over_ranks)
        prof = profile_read(lib, stream.cuda_stream)
        if tla.tla_last_device_status() != 0:
            raise RuntimeError(f"device status not OK after {w.name}")
        units = w.B * w.T * w.H
        rec = {"value": round(ws_n * w.B * w.T / (ms / 1e3), 1), "unit": "tokens/s",
               "ms": round(ms, 4), "steps": k,
               "config": {"B": w.B, "T": w.T, "H": w.H, "dk": w.dk, "dv": w.dv, "E": w.E,
                          "dtype": w.dtype, "delta_rule": w.use_delta,
                          "h0": f"N(0, {w.h0_std ** 2:g})" if w.h0_std else "zero",
                          "outputs": "fp32 o and final state"},
               "kernels": kernel_table(prof, w, units, peaks)}
        if w.dtype == "bf16":
            rec["s8d"] = s8d_roofline(w.E, w.dk, w.dv, False, units, ms, peaks)
            rec["l2"] = ("inputs and outputs larger than L2" if units * (2 * (2 * w.dk + w.dv) + 4 * w.dv)
                         > 129e6 else "working set within L2")
        else:
            rec["bound"] = "latency (tiny problem: one CTA per head and value block)"
        out[w.name] = rec
        del x, o, ht, fws
        torch.cuda.empty_cache()
    return out


def run_e2e(args, tla, x, w, dev, stream, o, fws, bws, grads, barrier, max_over_ranks, ws_n):
    """End to end through the public API with host buffers, as a training input pipeline
    runs it: every step copies its inputs from pinned host memory, runs forward and
    backward, and reads o and every gradient back into pinned host memory.  Three streams
    (host->device, compute, device->host) and two device copies of the inputs and outputs
    let step i's copies overlap the neighbouring steps' compute; the timed region runs from
    the first step's first upload to the last step's last download."""
    names = ["q", "k", "v", "q2", "k2", "g", "beta", "dO"]
    host_in = {n: x[n].cpu().pin_memory() for n in names}
    dev_in = [{n: torch.empty_like(x[n]) for n in names} for _ in range(2)]
    outs0 = {"o": o, **grads}
    outs = [outs0, {n: torch.empty_like(t) for n, t in outs0.items()}]
    host_out = {n: torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for n, t in outs0.items()}
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out.values())
    s_in, s_c, s_out = (torch.cuda.Stream(dev) for _ in range(3))
    ev = {k: [torch.cuda.Event() for _ in range(2)] for k in ("in_ready", "in_free", "out_ready", "out_free")}

    def step(i):
        j = i % 2
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(ev["in_free"][j])
            for n in names:
                dev_in[j][n].copy_(host_in[n], non_blocking=True)
            ev["in_ready"][j].record(s_in)
        with torch.cuda.stream(s_c):
            s_c.wait_event(ev["in_ready"][j])
            if i >= 2:
                s_c.wait_event(ev["out_free"][j])
            d = dev_in[j]
            og = outs[j]
            tla.tla_chunk_fwd(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], None,
                              use_delta=True, save_for_bwd=True, want_ht=False, o=og["o"],
                              workspace=fws)
            tla.tla_chunk_bwd(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["dO"], fws,
                              beta=d["beta"], use_delta=True, workspace=bws,
                              grads={n: t for n, t in og.items() if n != "o"})
            ev["in_free"][j].record(s_c)
            ev["out_ready"][j].record(s_c)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev["out_ready"][j])
            for n, t in og.items():
                host_out[n].copy_(t, non_blocking=True)
            ev["out_free"][j].record(s_out)

    for i in range(3):   # warm-up of the pipeline
        step(i)
    torch.cuda.synchronize()
    k = max(4, min(args.steps, 10))
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    for i in range(k):
        step(i)
    e1.record(s_out)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / k)
    return {"value": round(ws_n * w.B * w.T / (ms / 1e3), 1), "unit": "tokens/s",
            "ms_per_step": round(ms, 3), "steps": k, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "api": "paper_2609_36529_gb300.tla (ctypes -> libtla.so)",
            "pipeline": "3 streams (host->device, compute, device->host), 2 device copies of "
                        "inputs and outputs; every step uploads all inputs and downloads o "
                        "and every gradient"}


def run_packed(args, tla, inputs, w, dev, stream, barrier, max_over_ranks, ws_n, rank):
    """The headline step's tokens as packed documents (Appendix A, Kernels): one sequence of
    B*T tokens split into documents of log-normal length around 1000 tokens, each from its
    own zero state; forward + backward per step through the public API (cu_seqlens)."""
    total = w.B * w.T
    lens = inputs.packed_lengths(total, 1000, seed=rank)
    x, cu = inputs.packed_inputs(lens, w.H, w.dk, w.dv, w.E, dtype=w.dtype, backward=True,
                                 device=dev, seed=100 + rank)
    o = torch.empty(1, total, w.H, w.dv, dtype=OUT_DTYPE, device=dev)
    p = tla.make_problem(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], None, o,
                         None, use_delta=True, cu_seqlens=cu)
    fws = torch.empty(tla.fwd_workspace_bytes(p, True), dtype=torch.uint8, device=dev)
    bws = torch.empty(tla.bwd_workspace_bytes(p), dtype=torch.uint8, device=dev)
    grads = make_grads(x, OUT_DTYPE, dev)

    def step():
        tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], None,
                          use_delta=True, save_for_bwd=True, want_ht=False, o=o, workspace=fws,
                          cu_seqlens=cu)
        tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], fws,
                          beta=x["beta"], use_delta=True, workspace=bws, grads=grads,
                          cu_seqlens=cu)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    k = max(3, min(args.steps, 5))
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(k):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    if tla.tla_last_device_status() != 0:
        raise RuntimeError("device status not OK after the packed-document loop")
    ms = max_over_ranks(e0.elapsed_time(e1) / k)
    nc = sum((n + 63) // 64 for n in lens)
    return {"workload": f"gdn_fwdbwd_bf16_packed_T{total}_H{w.H}_d{w.dk}_E{w.E}",
            "value": round(ws_n * total / (ms / 1e3), 1), "unit": "tokens/s",
            "ms_per_step": round(ms, 4), "steps": k, "docs": len(lens),
            "doc_len": {"mean": round(total / len(lens), 1), "min": min(lens), "max": max(lens)},
            "chunks": nc, "chunks_uniform_batch": total // 64,
            "data": "synthetic; lengths log-normal around 1000 tokens (sigma 1), seeded"}


def _time_steps(step, k, warm, stream, barrier, max_over_ranks):
    for _ in range(warm):
        step()
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(k):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    return max_over_ranks(e0.elapsed_time(e1) / k)


def run_variants(args, tla, inputs, w, dev, stream, barrier, max_over_ranks, ws_n, rank,
                 headline):
    """Forward + backward tokens/s of the shape/gate variants: one log gate per head on the
    headline workload, the headline with o and the input gradients in bf16 (the input dtype),
    and on one 8192-token sequence the d_k vs E shapes of Table 4 at d_k E = 1024 (E = 8 with
    d_k = 128, E = 16 with d_k = 64) and E = 32 with d_k = 64.  Each case lists the kernels
    that ran (tensor-core `*_tc` or CUDA-core) and its state-update rate (tokens/s x E d_k d_v)
    against the headline's."""
    out = {}
    lib = tla.lib()
    cases = [("gate_per_head", w.B, w.T, w.H, w.dk, w.dv, w.E, True),
             ("bf16_outputs", w.B, w.T, w.H, w.dk, w.dv, w.E, False),
             ("E8_dk128", 1, w.T, w.H, 128, w.dv, 8, False),
             ("E16_dk64", 1, w.T, w.H, 64, w.dv, 16, False),
             ("E32_dk64", 1, w.T, w.H, 64, w.dv, 32, False)]
    for name, B, T, H, dk, dv, E, per_head in cases:
        out_dtype = torch.bfloat16 if name == "bf16_outputs" else OUT_DTYPE
        x = inputs.chunk_inputs(B, T, H, dk, dv, E, dtype=w.dtype, with_beta=True,
                                backward=True, device=dev, seed=200 + rank)
        if per_head:
            x["g"] = x["g"][..., 0].contiguous()
        o = torch.empty(B, T, H, dv, dtype=out_dtype, device=dev)
        p = tla.make_problem(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], None,
                             o, None, use_delta=True)
        fws = torch.empty(tla.fwd_workspace_bytes(p, True), dtype=torch.uint8, device=dev)
        bws = torch.empty(tla.bwd_workspace_bytes(p), dtype=torch.uint8, device=dev)
        grads = make_grads(x, out_dtype, dev)

        def step():
            tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], None,
                              use_delta=True, save_for_bwd=True, want_ht=False, o=o,
                              workspace=fws)
            tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], fws,
                              beta=x["beta"], use_delta=True, workspace=bws, grads=grads)

        ms = _time_steps(step, 3, 3, stream, barrier, max_over_ranks)
        val = ws_n * B * T / (ms / 1e3)
        lib.tla_profile_begin()   # one more step, untimed: which kernels ran
        step()
        torch.cuda.synchronize()
        kernels = sorted(profile_read(lib, stream.cuda_stream))
        out[name] = {"config": {"B": B, "T": T, "H": H, "dk": dk, "dv": dv, "E": E,
                                "gate": "per head [B,T,H]" if per_head else "per slice",
                                "outputs": "fp32" if out_dtype == torch.float32 else "bf16"},
                     "value": round(val, 1), "unit": "tokens/s", "ms_per_step": round(ms, 4),
                     "kernels": kernels,
                     "state_rate_vs_headline": round(val * E * dk * dv /
                                                     (headline * w.E * w.dk * w.dv), 4)}
        if B == w.B and T == w.T:
            out[name]["vs_headline"] = round(val / headline, 4)
        del x, fws, bws, grads, o
    if tla.tla_last_device_status() != 0:
        raise RuntimeError("device status not OK after the variant loops")
    return out


def run_layer_io(args, tla, inputs, w, dev, stream, barrier, max_over_ranks, rank, peaks):
    """The layer's input path and output gate (Algorithm 2) on the headline's token-heads
    (bf16 projection output, K = 4 convolution, fp32 operator output and gradients): device
    time per call and algorithmic bytes (each tensor read or written once) per second."""
    B, T, H, dk, dv, E, K = w.B, w.T, w.H, w.dk, w.dv, w.E, 4
    x = inputs.layer_inputs(B, T, H, dk, dv, E, K, dtype=w.dtype, device=dev, seed=300 + rank)
    args_p = [x[n] for n in ("P", "conv_w", "gate_in", "gate_bias", "A_log", "beta_in")]
    gen = torch.Generator(dev).manual_seed(301 + rank)
    grads = {n: torch.randn(B, T, H, c, device=dev, generator=gen)
             for n, c in (("dq", dk), ("dk", dk), ("dv", dv), ("dq2", E), ("dk2", E), ("dg", E))}
    grads["dbeta"] = torch.randn(B, T, H, device=dev, generator=gen)
    dy = torch.randn(B, T, H, dv, device=dev, generator=gen).to(x["z"].dtype)
    units = B * T * H
    C = 2 * dk + dv + 2 * E
    eb = 2 if w.dtype == "bf16" else 4
    bytes_per = {   # per token-head, every tensor touched once
        "prologue_fwd": C * eb + E * 4 + 4 + C * eb + E * 4 + 4,
        "prologue_bwd": C * eb + (2 * dk + dv + 2 * E) * 4 + E * 4 + 4 + E * 4 + 4 + C * eb + E * 4 + 4,
        "gate_fwd": dv * 4 + dv * eb + dv * eb,
        "gate_bwd": dv * 4 + 2 * dv * eb + dv * 4 + dv * eb}
    calls = {"prologue_fwd": lambda: tla.layer_prologue(*args_p, dk, dv, E),
             "prologue_bwd": lambda: tla.layer_prologue_bwd(*args_p, dk, dv, E, grads),
             "gate_fwd": lambda: tla.output_gate(x["o"], x["z"], x["w_norm"]),
             "gate_bwd": lambda: tla.output_gate_bwd(x["o"], x["z"], x["w_norm"], dy)}
    peak = peaks["hbm_gbs"]
    out = {"workload": f"layer_io_B{B}_H{H}_T{T}_d{dk}_E{E}_K{K}", "unit": "GB/s", "peak": peak,
           "peak_source": "hbm copy bandwidth, " + peaks["source"]}
    for name, fn in calls.items():
        ms = _time_steps(fn, 3, 3, stream, barrier, max_over_ranks)
        gbs = bytes_per[name] * units / (ms / 1e3) / 1e9
        out[name] = {"ms": round(ms, 4), "achieved_gbs": round(gbs, 1), "frac": round(gbs / peak, 4),
                     "bytes_per_token_head": bytes_per[name]}
    del x, args_p, grads, dy
    torch.cuda.empty_cache()
    # the input projection GEMM with the input path fused into its epilogue, at the paper's
    # 1.3B-parameter width (d_model 2048, 16 heads of d = 128): tensor-bound
    Dm = 2048
    xp = inputs.projection_inputs(B, T, H, dk, dv, E, Dm, K, device=dev, seed=310 + rank)
    C = 2 * dk + dv + 2 * E
    call = lambda: tla.layer_projection(xp["u"], xp["W"], xp["conv_w"], xp["gate_in"],  # noqa: E731
                                        xp["gate_bias"], xp["A_log"], xp["beta_in"], dk, dv, E)
    ms = _time_steps(call, 3, 3, stream, barrier, max_over_ranks)
    flops = 2.0 * B * T * Dm * H * C
    tf = flops / (ms / 1e3) / 1e12
    out["projection"] = {"ms": round(ms, 4), "tflops": round(tf, 1),
                         "peak_tflops": peaks["bf16_tflops"],
                         "frac": round(tf / peaks["bf16_tflops"], 4),
                         "bound": "tensor", "d_model": Dm, "channels_per_head": C,
                         "algorithmic_flops": flops,
                         "peak_source": "bf16 dense burst, " + peaks["source"],
                         "what": "u W^T (bf16, fp32 accumulation) + causal conv K=4, SiLU/softplus, "
                                 "L2 norms, log gates, beta in the epilogue; q,k,v,q',k' bf16 out"}
    return out


def run_decode(args, tla, inputs, dev, stream, lib, peaks, barrier, max_over_ranks, ws_n):
    dw = inputs.DECODE
    if args.decode_batch:   # profiling option: fewer sequences of the same shape
        dw = dataclasses.replace(dw, B=args.decode_batch, name=f"{dw.name}_batch{args.decode_batch}")
    gen = torch.Generator(dev)
    gen.manual_seed(1000 + dist_env()[1])
    state = torch.empty(dw.B, dw.H, dw.E, dw.dk, dw.dv, dtype=torch.float32, device=dev)
    res = {}
    for variant, use_delta in (("sgla", False), ("gdn", True)):
        pre = inputs.chunk_inputs(dw.B, dw.prefill, dw.H, dw.dk, dw.dv, dw.E, dtype="bf16",
                                  with_beta=True, device=dev, gen=gen)
        ws = None
        _, _, ws = tla.tla_chunk_fwd(pre["q"], pre["k"], pre["v"], pre["q2"], pre["k2"], pre["g"],
                                     pre["beta"], None, use_delta=use_delta, save_for_bwd=False,
                                     ht=state)
        del pre, ws
        steps = [inputs.decode_inputs(dw.B, dw.H, dw.dk, dw.dv, dw.E, dtype="bf16", device=dev,
                                      gen=gen) for _ in range(dw.steps)]
        o = torch.empty(dw.B, dw.H, dw.dv, dtype=torch.bfloat16, device=dev)
        # warm-up launches on a one-sequence scratch state keep the measured sequence intact
        scratch = state[:1].clone()
        for s in steps[:3]:
            tla.tla_decode_step(scratch, *(s[n][:1].contiguous() for n in
                                           ("q", "k", "v", "q2", "k2", "g", "beta")),
                                use_delta=use_delta)
        del scratch
        torch.cuda.synchronize()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        lib.tla_profile_begin()
        e0.record(stream)
        for s in steps:
            tla.tla_decode_step(state, s["q"], s["k"], s["v"], s["q2"], s["k2"], s["g"], s["beta"],
                                use_delta=use_delta, o=o)
        e1.record(stream)
        torch.cuda.synchronize()
        prof = profile_read(lib, stream.cuda_stream)
        ms = max_over_ranks(e0.elapsed_time(e1) / dw.steps)
        kern_ms = prof["decode_step"]["ms"] / prof["decode_step"]["launches"]
        bytes_step = 8.0 * dw.E * dw.dk * dw.dv * dw.B * dw.H
        gbs = bytes_step / (kern_ms / 1e3) / 1e9
        res[variant] = {"ms_per_step": round(ms, 4), "kernel_ms": round(kern_ms, 4),
                        "seq_steps_per_s": round(ws_n * dw.B / (ms / 1e3), 1),
                        "achieved_gbs": round(gbs, 1), "frac": round(gbs / peaks["hbm_gbs"], 4),
                        "launches": prof["decode_step"]["launches"]}
        del steps
    return {"workload": dw.name, "unit": "GB/s", "bound": "hbm", "peak": peaks["hbm_gbs"],
            "peak_source": f"hbm copy bandwidth, {peaks['source']}",
            "bytes_per_step": 8 * dw.E * dw.dk * dw.dv * dw.B * dw.H,
            "traffic": ncu_traffic("decode_step", dw.B * dw.H),
            "state": "fp32 [256,32,8,128,128] (4.3 GB, larger than L2)", "inputs": "bf16",
            **res}


def oracle_baseline(x, w, seconds_target=15.0, T_sample=None):
    """Time the float64 oracle (fwd+bwd) on a sample of whole heads on this host's cores."""
    import oracle
    cores = oracle.num_threads()
    T = T_sample or w.T
    nh = max(1, min(cores, w.B * w.H))
    picks = [(i // w.H, i % w.H) for i in range(nh)]

    def sel(t, per_token=True):
        return torch.stack([t[b, :T, h] for b, h in picks])[:, :, None].double().cpu().numpy()

    c = {n: sel(x[n]) for n in ("q", "k", "v", "q2", "k2", "g", "beta", "dO")}
    t0 = time.perf_counter()
    oracle.forward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["beta"], None)
    oracle.backward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["dO"], c["beta"], None)
    dt = time.perf_counter() - t0
    tokens_equiv = nh * T / w.H   # one token = all H heads of one position
    return {"value": round(tokens_equiv / dt, 3), "unit": "tokens/s", "cores": cores,
            "kind": "oracle", "seconds": round(dt, 2),
            "sample": f"{nh} whole heads (b,h) x {T} tokens of {w.name}, float64 token "
                      f"recurrence forward + backward, OpenMP over heads; tokens/s counts "
                      f"{nh}/{w.H} of a position's heads as {nh / w.H:.3f} tokens"}


# ----------------------------------------------------------------------------- reference arm

def run_reference(args):
    ws_n, rank, _ = dist_env()
    if rank != 0:
        return
    from paper_2609_36529_gb300 import inputs
    import oracle
    w = inputs.GDN_FWDBWD_BF16
    cores = oracle.num_threads()
    nh = max(1, min(cores, w.B * w.H))
    T = args.ref_tokens
    x = inputs.chunk_inputs(1, T, nh, w.dk, w.dv, w.E, dtype="bf16", with_beta=True,
                            backward=True, device="cpu", seed=0)
    c = {n: x[n].double().numpy() for n in ("q", "k", "v", "q2", "k2", "g", "beta", "dO")}

    def step():
        oracle.forward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["beta"], None)
        oracle.backward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["dO"], c["beta"], None)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = (time.perf_counter() - t0) / args.steps
    tokens_equiv = nh * T / w.H
    value = tokens_equiv / dt
    sample = (f"{nh} heads x {T} tokens per step (shape of {w.name}: d_k=d_v={w.dk}, E={w.E}), "
              f"float64 oracle forward + backward on {cores} host threads; tokens/s counts "
              f"{nh}/{w.H} of a position's heads as {nh / w.H:.3f} tokens")
    line = {"metric": HEADLINE_METRIC, "value": round(value, 3), "unit": "tokens/s",
            "n_gpus": ws_n, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(dt * 1e3, 2), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "T": w.T, "H": w.H, "dk": w.dk, "dv": w.dv,
                       "E": w.E, "chunk": CHUNK, "variant": "triadic GDN (joint-key delta rule)"},
            "impl": "reference",
            "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-packed", action="store_true")
    ap.add_argument("--no-variants", action="store_true")
    ap.add_argument("--no-layer", action="store_true")
    ap.add_argument("--no-fwd-workloads", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--ref-tokens", type=int, default=1024,
                    help="tokens per head in one reference-arm step")
    ap.add_argument("--batch", type=int, default=0,
                    help="profiling only: run B sequences instead of the workload's 8")
    ap.add_argument("--fwd-only", action="store_true",
                    help="profiling only: time the forward alone (not the headline metric)")
    ap.add_argument("--decode-batch", type=int, default=0,
                    help="profiling only: decode workload with this many sequences")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        print("bench: at least 3 warm-up steps are required; using 3", file=sys.stderr)
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
